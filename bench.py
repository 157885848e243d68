"""Benchmark: the exact parallelism search on the 70B-like heterogeneous
workload (L=80 layers, S=8 stages, M=32, 3 device types, TP in {1,2,4,8}),
one poseidon_search call per step through the C ABI.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line.  `value` = DAG makespan evaluations per second of
search (device time, CUDA events around each step, L2 flushed between
steps); `time_to_plan_s` = mean step time.  `--impl reference` times the
CPU oracle on a bounded sample of the same workload instead.
With torchrun (N > 1) every rank runs an independent replica of the search
(weak scaling); the step time is the maximum over ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import gen  # noqa: E402

WORKLOAD = ("70B-like search: L=80, S=8, M=32, 3 device types (312/125/65 TFLOPS, "
            "80/32/16 GB, 32/32/64 devices), TP in {1,2,4,8}, D=16/t, stage-type counts "
            "(2,2,4): 1680 slices, 4.87e12 plans")
METRIC = "DAG makespan evals/sec (time-to-optimal plan at L=80, S=8)"
WARMUP_SAMPLES = 500  # the paper's warm-up count (Sec. 4.2.3)
SM_LANES = 128  # INT32 lanes per SM (4 partitions x 32)
ENTRY_BYTES = 32  # one frontier entry / one complete plan
# DRAM bytes per evaluated plan of leaf_kernel, from one ncu capture of
# dram__bytes_read.sum + dram__bytes_write.sum over a config-4 search's leaf
# launches (the leaf kernel's ncu summary), valid while the kernel's
# sources hash to LEAF_SOURCES_SHA256 (else the traffic is reported as null)
LEAF_DRAM_BYTES_PER_PLAN = 59682816 / 1925970
LEAF_SOURCES = ("paper_2609_06086_gb300/csrc/search_kernels.cuh",
                "paper_2609_06086_gb300/csrc/common.cuh")
LEAF_SOURCES_SHA256 = "c701e85b0c1184ee"
PRUNE_NAMES = {1: "stage-level, Eq. 2 as printed (Theorem 1)",
               2: "stage-level, tightened: Eq. 2 with P2P edges + completion bounds"}


def measured_hbm():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        return float(json.load(open(path))["hbm_gbs"]), "measured copy bandwidth (MEASURED_PEAKS.json)"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback 6.8 TB/s (MEASURED_PEAKS.json absent)"


def leaf_sources_unchanged() -> bool:
    import hashlib
    h = hashlib.sha256()
    for f in LEAF_SOURCES:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16] == LEAF_SOURCES_SHA256


def dist_env():
    return int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")), \
        int(os.environ.get("LOCAL_RANK", "0"))


class Clocks:
    """nvidia-smi sampling during the timed region."""

    def __init__(self, index):
        self.proc = None
        self.path = os.path.join(tempfile.gettempdir(), f"poseidon_clocks_{os.getpid()}.csv")
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        self.index, self.query = index, q
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(index), f"--query-gpu={q}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if not self.proc:
            return None
        self.proc.terminate()
        self.proc.wait()
        self.f.close()
        if not any(len(line.split(",")) >= 9 for line in open(self.path)):
            # a timed region shorter than the sampling period: one reading
            # taken as it ends
            try:
                with open(self.path, "a") as f:
                    subprocess.run(["nvidia-smi", "-i", str(self.index),
                                    f"--query-gpu={self.query}", "--format=csv,noheader,nounits"],
                                   stdout=f, stderr=subprocess.DEVNULL, timeout=10)
            except (OSError, subprocess.SubprocessError):
                pass
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            p = [x.strip() for x in line.split(",")]
            if len(p) < 9:
                continue
            try:
                sm.append(float(p[1]))
                mx = max(mx, float(p[2]))
            except ValueError:
                continue
            for n, v in zip(names, p[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def oracle_sample_rate(seconds: float, seed: int = 0):
    """The CPU oracle (single thread, as it stands) evaluating config-4-shaped
    plans (S=8, M=32, TP index 3) until `seconds` have elapsed."""
    import oracle
    w = gen.config4()
    tab = oracle.OracleTables.from_workload(w)
    c = gen.random_candidates(4096, L=w.L, n_types=3, S_range=(8, 8), M_range=(32, 32),
                              seed=seed)
    c["tp_idx"] = 3
    n, t0 = 0, time.perf_counter()
    while time.perf_counter() - t0 < seconds:
        oracle.eval_batch(tab, c[:512])
        n += 512
    dt = time.perf_counter() - t0
    return n / dt, n, dt


def _oracle_worker(args):
    seconds, seed = args
    return oracle_sample_rate(seconds, seed)


def oracle_all_cores_rate(seconds: float):
    """The same single-threaded oracle in one process per host core (spawned,
    so no CUDA state is inherited), each on its own sample for `seconds`;
    returns (summed evals/s, processes, evaluations)."""
    import multiprocessing as mp
    n = max(1, os.cpu_count() or 1)
    with mp.get_context("spawn").Pool(n) as pool:
        res = pool.map(_oracle_worker, [(seconds, 100 + i) for i in range(n)])
    return sum(r[0] for r in res), n, sum(r[1] for r in res)


def _oracle_search_part(args):
    cfg, part, n_parts = args
    import oracle
    w = gen.get_config(cfg)
    plan, st = oracle.search(w, prune=True, warmup=500, seed=0, part=part, n_parts=n_parts)
    return plan, st["leaves_evaluated"] + st["warmup_evaluated"]


def oracle_time_to_plan(configs_procs):
    """The CPU oracle's search (Eq. 2 prune as printed, 500 warm-up samples,
    the paper's method) on each (config, processes): the slices are dealt
    round-robin to `processes` spawned single-threaded oracle processes
    (orc_search_part), the best plan of the parts by (T/(D*M), global index)
    is the result; wall time from the first part's start to the last part's
    end (the process pool is started before the clock)."""
    import multiprocessing as mp
    from fractions import Fraction
    n_max = max(n for _, n in configs_procs)
    out = []
    with mp.get_context("spawn").Pool(n_max) as pool:
        pool.map(_oracle_worker, [(0.01, i) for i in range(n_max)])  # workers up, oracle loaded
        for cfg, n in configs_procs:
            t0 = time.perf_counter()
            res = pool.map(_oracle_search_part, [(cfg, i, n) for i in range(n)])
            wall = time.perf_counter() - t0
            best = None
            for plan, _ in res:
                if plan["found"]:
                    key = (Fraction(plan["T"], plan["D"] * plan["M"]), plan["global_index"])
                    if best is None or key < best[0]:
                        best = (key, plan)
            out.append({"config": cfg, "seconds": round(wall, 3), "processes": n,
                        "evaluations": sum(e for _, e in res),
                        "T_us": best[1]["T"] if best else None,
                        "global_index": best[1]["global_index"] if best else None})
    return out


def _oracle_eval_chunk(args):
    lo, hi = args
    import oracle
    w = gen.config5_tables()
    tab = oracle.OracleTables.from_workload(w)
    c = gen.config5_candidates(hi, seed=0)[lo:hi]
    t0 = time.perf_counter()
    oracle.eval_batch(tab, c)
    return hi - lo, time.perf_counter() - t0


def oracle_config5_rate(n, procs):
    """The CPU oracle evaluating the first n candidates of the config-5 batch
    (L=64, S~U{2..16}, M~U{8..128}), split into `procs` spawned
    single-threaded processes; evals/s = n / the slowest process's time."""
    import multiprocessing as mp
    step = (n + procs - 1) // procs
    with mp.get_context("spawn").Pool(procs) as pool:
        res = pool.map(_oracle_eval_chunk, [(i * step, min(n, (i + 1) * step))
                                            for i in range(procs) if i * step < n])
    return n / max(t for _, t in res), max(t for _, t in res)


def eval_throughput(P, torch, n, reps, peak_alu, schedule=0, space=None):
    """poseidon_eval_batch on n config-5 candidates (L=64, S ~ U{2..16},
    M ~ U{8..128}, 2 device types), device-resident, timed with CUDA events
    on the launching stream; inputs (16 B x n) exceed L2 for n >= 1e7.
    Under Interleaved 1F1B (schedule 2) the records are the interleaved
    sweep on the same tables: N ~ U{1..8} devices, V ~ U{2..16//N} chunks,
    M ~ U{8..128} rounded down to a multiple of N; S counts the N*V virtual
    stages below."""
    w = gen.config5_tables() if space is None else space
    if space is not None:
        c = gen.search_space_sample(space, n, seed=0)
        S = c["S"].astype(np.int64)
    elif schedule == 2:
        c = gen.interleaved_candidates(n, L=w.L, seed=0)
        S = c["S"].astype(np.int64) * c["V"].astype(np.int64)
    else:
        c = gen.config5_candidates(n, seed=0)
        S = c["S"].astype(np.int64)
    M = c["M"].astype(np.int64)
    relax = int((2 * S * M).sum())
    ops = 3 * relax + 11 * int(S.sum())  # 6SM + 11S integer ops per candidate
    h = P.Handle(P.Tables.from_workload(w), schedule=schedule)
    d_c = torch.from_numpy(c.view(np.uint8)).cuda()
    del c
    d_T = torch.empty(n, dtype=torch.int32, device="cuda")
    d_F = torch.empty(n, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()
    for _ in range(2):
        P.poseidon_eval_batch(h, d_c.data_ptr(), n, d_T.data_ptr(), d_F.data_ptr(),
                              stream.cuda_stream)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    ms = 0.0
    for _ in range(reps):
        ev0.record(stream)
        P.poseidon_eval_batch(h, d_c.data_ptr(), n, d_T.data_ptr(), d_F.data_ptr(),
                              stream.cuda_stream)
        ev1.record(stream)
        torch.cuda.synchronize()
        ms += ev0.elapsed_time(ev1)
    sec = ms / 1e3 / reps
    h.close()
    ach = ops / sec / 1e12
    return {"workload": (f"{space.name}: uniform sample of the whole search space "
                         "(no memory cut, no prune)" if space is not None else
                         "interleaved sweep: L=64, N~U{1..8}, V~U{2..16/N}, M~U{8..128} "
                         "(multiple of N), 2 device types" if schedule == 2 else
                         "config 5: L=64, S~U{2..16}, M~U{8..128}, 2 device types"),
            "schedule": ["1F1B", "Eager 1F1B", "Interleaved 1F1B"][schedule],
            "batch": n, "ms_per_call": round(sec * 1e3, 4), "evals_per_s": n / sec,
            "relaxations_per_s": relax / sec, "bound": "alu", "achieved": round(ach, 3),
            "unit": "Tops/s", "peak": round(peak_alu, 3), "frac": round(ach / peak_alu, 4)}


def run_reference(args, rank, world):
    if rank != 0:
        return
    # each step a bounded sample, so that the whole run stays near two minutes
    per_step = max(0.05, min(2.0, 120.0 / max(1, args.steps)))
    for _ in range(args.warmup):
        oracle_sample_rate(0.2)
    rates, total_n, total_t = [], 0, 0.0
    for k in range(args.steps):
        r, n, dt = oracle_sample_rate(per_step, seed=k)
        rates.append(r)
        total_n += n
        total_t += dt
    value = total_n / total_t
    sample = (f"{total_n} config-4 plan evaluations (S=8, M=32, L=80) by the single-threaded "
              f"CPU oracle, {per_step:.2f} s per step")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "evals/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * total_t / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int32", "data": "synthetic",
        "config": {"workload": WORKLOAD, "sample": sample},
        "cpu_baseline": {"value": value, "unit": "evals/s", "cores": 1, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "evals/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


def run_ours(args, rank, world, local_rank):
    import torch
    import paper_2609_06086_gb300 as P

    torch.cuda.set_device(local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if args.backend == "nccl" else "gloo")
    w = gen.config4()
    prob, keep = P.make_problem(w, warmup=WARMUP_SAMPLES, prune=args.prune, seed=0,
                                frontier_cap=args.frontier_cap)
    # the same search with CUDA events around every kernel, for the per-kernel
    # breakdown (run after the timed steps; the events cost host time)
    prob_prof, keep_prof = P.make_problem(w, warmup=WARMUP_SAMPLES, prune=args.prune, seed=0,
                                          frontier_cap=args.frontier_cap, profile=True)
    tab_bytes = sum(a.nbytes for a in keep[0].arrays.values()) + sum(a.nbytes for a in keep[1:])
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.int32, device="cuda")

    for _ in range(args.warmup):
        P.poseidon_search(prob)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    clocks = Clocks(torch.cuda.current_device()) if rank == 0 else None
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    dev_ms, wall_ms, plans = [], [], []
    agg = dict(evaluated=0, warmup_evaluated=0, relaxations=0, launches=0, ms_expand=0.0, ms_complete=0.0,
               ms_leaf=0.0, expand_launches=0, complete_launches=0, leaf_launches=0,
               parents_expand=0, parents_complete=0, leaves=0, prefixes=0,
               ms_setup=0.0, ms_warmup=0.0, ms_search=0.0)
    # the device time brackets the library call alone (the binding's plan and
    # statistics dicts are built after ev1); e2e times the public Python call
    Lib, Cb = P.lib(), P.binding.C
    plan_c, st_c = P.binding.pos_plan(), P.binding.pos_search_stats()

    def timed_search_call(pr):
        """One search with L2 flushed before it; the CUDA events bracket the
        library call alone.  Returns (ms, plan dict, stats dict)."""
        pc, sc = P.binding.pos_plan(), P.binding.pos_search_stats()
        flush.zero_()
        torch.cuda.synchronize()
        ev0.record()
        rc_ = Lib.poseidon_search(Cb.byref(pr), Cb.byref(pc), Cb.byref(sc))
        ev1.record()
        torch.cuda.synchronize()
        if rc_ != P.binding.POS_OK:
            raise P.PoseidonError(rc_, Lib.poseidon_last_error().decode())
        return ev0.elapsed_time(ev1), P.binding.plan_dict(pr, pc), P.binding.stats_dict(sc)

    for _ in range(args.steps):
        flush.zero_()  # evict L2 (129 MB) between steps
        torch.cuda.synchronize()
        ev0.record()
        rc = Lib.poseidon_search(Cb.byref(prob), Cb.byref(plan_c), Cb.byref(st_c))
        ev1.record()
        torch.cuda.synchronize()
        if rc != P.binding.POS_OK:
            raise P.PoseidonError(rc, Lib.poseidon_last_error().decode())
        dev_ms.append(ev0.elapsed_time(ev1))
        plans.append(P.binding.plan_dict(prob, plan_c))
        st = P.binding.stats_dict(st_c)
        for k in agg:
            agg[k] += st[k]
    for _ in range(args.steps):
        flush.zero_()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        P.poseidon_search(prob)
        torch.cuda.synchronize()
        wall_ms.append(1e3 * (time.perf_counter() - t0))
    clk = clocks.stop() if clocks else None
    # per-kernel breakdown: the same number of steps again, with CUDA events
    # around every launch on the library's stream (profile=1)
    prof_ms = []
    kagg = {k: 0 for k in agg}
    for k in ("ms_depth", "launches_depth", "parents_depth", "children_depth"):
        kagg[k] = [0] * 16
    for _ in range(args.steps):
        ms_, plan_p, st_p = timed_search_call(prob_prof)
        prof_ms.append(ms_)
        for k in kagg:
            if isinstance(kagg[k], list):
                kagg[k] = [u + v for u, v in zip(kagg[k], st_p[k])]
            else:
                kagg[k] += st_p[k]
    t_dev = sum(dev_ms)
    if dist:
        tt = torch.tensor([t_dev], dtype=torch.float64,
                          device="cuda" if args.backend == "nccl" else "cpu")
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        t_dev = float(tt.item())
        dist.barrier()
    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return
    import json as _json
    ref = _json.load(open(os.path.join(ROOT, "tests", "golden", "search_plans.json")))["config4"]
    parity = all(p["global_index"] == ref["plan"]["global_index"] and p["T"] == ref["plan"]["T"]
                 for p in plans)
    evals = agg["evaluated"] * world
    value = evals / (t_dev / 1e3)
    e2e = evals / (sum(wall_ms) / 1e3)
    props = torch.cuda.get_device_properties(torch.cuda.current_device())
    n_sm = props.multi_processor_count
    # Per kernel (device time from CUDA events around every launch on the
    # library's stream, profiled steps): the leaf kernel (makespans of the
    # complete plans) and the level kernel of each parent depth x (x = S-2
    # completes the last two stages).  Algorithmic work per unit:
    #  leaf    : int32 ops, 3 per DAG node relaxation + 9 per stage
    #  level x : bytes, a 32-byte frontier entry read per parent and a 32-byte
    #            child (or complete plan) written per child
    mhz = (clk or {}).get("sm_mhz") or 2070.0
    peak_alu = n_sm * SM_LANES * mhz * 1e6 / 1e12  # Tops/s at the measured SM clock
    # the relaxation microbenchmark: does the GPU run max/add at that rate?
    p_ops, p_ms = P.binding.poseidon_int32_probe(torch.cuda.current_stream().cuda_stream)
    probe = {"tops": round(p_ops / (p_ms / 1e3) / 1e12, 3),
             "frac_of_nominal": round(p_ops / (p_ms / 1e3) / 1e12 / peak_alu, 4),
             "what": "max(pred + edge, clock) + weight in 8 independent chains per thread, "
                     "8 blocks of 256 threads per SM"}
    peak_hbm, hbm_src = measured_hbm()
    S = w.S
    kinds, launches, work, bound = {}, {}, {}, {}
    kinds["leaf_kernel"] = kagg["ms_leaf"]
    launches["leaf_kernel"] = kagg["leaf_launches"]
    # the timed leaf launches are the search's (the warm-up's are not in ms_leaf)
    leaf_plans = kagg["evaluated"] - kagg["warmup_evaluated"]
    work["leaf_kernel"] = (3 * 2 * S * w.M_list[0] + 9 * S) * leaf_plans
    bound["leaf_kernel"] = ("alu", "Tops/s", peak_alu, 1e12)
    for x in range(S - 1):
        name = f"level_kernel<{'complete' if x == S - 2 else 'expand'}, depth {x}>"
        kinds[name] = kagg["ms_depth"][x]
        launches[name] = kagg["launches_depth"][x]
        work[name] = ENTRY_BYTES * (kagg["parents_depth"][x] + kagg["children_depth"][x])
        bound[name] = ("hbm", "GB/s", peak_hbm, 1e9)
    dom = max(kinds, key=kinds.get)
    per_kind = {}
    for k in kinds:
        b, unit, peak, scale = bound[k]
        ach = work[k] / max(kinds[k] / 1e3, 1e-12) / scale
        per_kind[k] = {"ms_per_step": round(kinds[k] / args.steps, 4),
                       "launches_per_step": launches[k] / args.steps, "bound": b,
                       "achieved": round(ach, 3), "unit": unit, "frac": round(ach / peak, 4)}
    b, unit, peak, scale = bound[dom]
    traffic = None
    if dom == "leaf_kernel" and leaf_sources_unchanged():
        traffic = round(LEAF_DRAM_BYTES_PER_PLAN * leaf_plans / max(1, launches[dom]))
    roof = {"bound": b, "kernel": dom, "unit": unit, "peak": round(peak, 3),
            "achieved": per_kind[dom]["achieved"], "frac": per_kind[dom]["frac"],
            "work_per_launch": work[dom] / max(1, launches[dom]), "traffic": traffic,
            "traffic_note": ("DRAM bytes per launch: ncu dram__bytes_read.sum + "
                             "dram__bytes_write.sum per plan (one ncu capture of a config-4 search) "
                             "x plans per launch" if traffic is not None else None),
            "peak_note": (f"{n_sm} SMs x {SM_LANES} int32 lanes x {mhz:.0f} MHz (median SM "
                          "clock under load)" if b == "alu" else hbm_src)}
    if b == "alu":
        # the relaxation microbenchmark runs above the lane count (fused
        # add-max): the fraction of that measured rate, beside the nominal one
        roof["peak_measured"] = probe["tops"]
        roof["frac_of_measured"] = round(roof["achieved"] / probe["tops"], 4)
    evals = [eval_throughput(P, torch, int(n), 5, peak_alu) for n in args.eval_sizes]
    for e in evals:
        e["frac_of_measured"] = round(e["achieved"] / probe["tops"], 4)
    # batch-size sweep of the same evaluator (config 5)
    sweep = []
    for n in args.eval_sweep:
        e = eval_throughput(P, torch, int(n), 5, peak_alu)
        sweep.append({k: e[k] for k in ("batch", "ms_per_call", "evals_per_s",
                                         "relaxations_per_s", "achieved", "frac")})
    evals_eager = [eval_throughput(P, torch, int(n), 5, peak_alu, schedule=1)
                   for n in args.eval_sizes[:1]]
    evals_il = [eval_throughput(P, torch, int(n), 5, peak_alu, schedule=2)
                for n in args.eval_sizes[:1]]
    # config 3 unpruned: a uniform sample of its 4.4e9-plan space through the
    # evaluator (S = 8, M = 64: 1024 relaxations per plan)
    evals_c3 = [eval_throughput(P, torch, int(n), 5, peak_alu, space=gen.config3())
                for n in args.eval_sizes[:1]]
    # the same search under Eager 1F1B (App. B schedule), for comparison
    ref_e = _json.load(open(os.path.join(ROOT, "tests", "golden", "search_plans.json")))
    ref_e = ref_e.get("config4_eager", {}).get("plan", {})
    prob_e, keep_e = P.make_problem(w, warmup=WARMUP_SAMPLES, prune=args.prune, seed=0,
                                    frontier_cap=args.frontier_cap, schedule=1)
    P.poseidon_search(prob_e)
    e_ms, e_ev, e_ok = [], 0, True
    for _ in range(max(3, min(100, args.steps // 2))):
        ms_, plan_e, st_e = timed_search_call(prob_e)
        e_ms.append(ms_)
        e_ev += st_e["evaluated"]
        e_ok &= plan_e["global_index"] == ref_e.get("global_index")
    # layer-level (ridge) pruning, Theorem 2: value against the exact optimum
    ridge_lines = []
    for sched, exact_ms, exact_T in ((0, t_dev / args.steps, plans[-1]["T"]),
                                     (1, sum(e_ms) / len(e_ms), plan_e["T"])):
        prob_r, keep_r = P.make_problem(w, warmup=WARMUP_SAMPLES, prune=args.prune, seed=0,
                                        frontier_cap=args.frontier_cap, schedule=sched,
                                        ridge=True)
        P.poseidon_search(prob_r)
        r_ms = []
        for _ in range(max(3, min(100, args.steps // 2))):
            ms_, plan_r, st_r = timed_search_call(prob_r)
            r_ms.append(ms_)
        ridge_lines.append({"schedule": "Eager 1F1B" if sched else "1F1B",
                            "time_to_plan_s": sum(r_ms) / len(r_ms) / 1e3,
                            "speedup_vs_exact": exact_ms / (sum(r_ms) / len(r_ms)),
                            "T_us": plan_r["T"], "exact_T_us": exact_T,
                            "same_value": plan_r["T"] == exact_T,
                            "evaluations_per_step": st_r["evaluated"],
                            "pruned_by_ridge": st_r["pruned_ridge"]})
    eager_search = {"schedule": "Eager 1F1B", "prune": PRUNE_NAMES[args.prune],
                    "time_to_plan_s": sum(e_ms) / len(e_ms) / 1e3,
                    "evaluations_per_step": e_ev / len(e_ms), "T_us": plan_e["T"],
                    "matches_oracle": e_ok}
    # the search with a TP degree chosen per stage (POS_PLACE_DEVICES): config
    # 4's tables and cluster, D in {2, 4, 8, 16}, each type's devices used up
    def timed_search(wl, ref_plan, **kw):
        pr, kp = P.make_problem(wl, warmup=WARMUP_SAMPLES, seed=0,
                                frontier_cap=args.frontier_cap, **kw)
        P.poseidon_search(pr)
        ms, ok, st_sum = [], True, 0
        for _ in range(max(3, min(100, args.steps // 2))):
            ms_, pl, st_ = timed_search_call(pr)
            ms.append(ms_)
            st_sum += st_["evaluated"]
            ok &= ref_plan is not None and all(pl[k] == ref_plan.get(k) for k in
                                               ("global_index", "T", "layers"))
        return pl, st_, sum(ms) / len(ms), st_sum / len(ms), ok

    stored = _json.load(open(os.path.join(ROOT, "tests", "golden", "search_plans.json")))
    w_ps = gen.config4_per_stage_tp()
    ref_ps = stored.get("config4_per_stage_tp", {}).get("plan")
    pl_ps, st_ps, ms_ps, ev_ps, ok_ps = timed_search(w_ps, ref_ps, prune=args.prune)
    per_stage_tp = {"workload": w_ps.name, "prune": PRUNE_NAMES[args.prune],
                    "time_to_plan_s": ms_ps / 1e3, "evaluations_per_step": ev_ps,
                    "slices": st_ps["slices"], "slices_feasible": st_ps["slices_feasible"],
                    "host_ms": {k: round(st_ps[k], 3) for k in ("ms_setup", "ms_warmup",
                                                                 "ms_search")},
                    "plan": {"T_us": pl_ps["T"], "D": pl_ps["D"], "tp_per_stage":
                             [w_ps.tp_list[i] for i in pl_ps["tps"]], "types": pl_ps["types"],
                             "layers": pl_ps["layers"]},
                    "matches_oracle": ok_ps}
    # the search over Interleaved 1F1B plans (config 2 tables, V = 2 and 3
    # chunks per device), against the oracle's stored plans
    il_lines = []
    for V in (2, 3):
        ref_il = stored.get(f"config2_il_v{V}", {}).get("plan")
        pl_il, st_il, ms_il, ev_il, ok_il = timed_search(gen.config2(), ref_il,
                                                          prune=args.prune, schedule=2, V=V)
        il_lines.append({"workload": "config 2 (L=32, S=4, M in {8,16,32}), V = %d" % V,
                         "prune": PRUNE_NAMES[args.prune], "time_to_plan_s": ms_il / 1e3,
                         "evaluations_per_step": ev_il, "T_us": pl_il["T"],
                         "matches_oracle": ok_il})
    # the other stage-level prune, same workload, for comparison (not the headline)
    other = PRUNE_NAMES[1 if args.prune == 2 else 2]
    other_mode = 1 if args.prune == 2 else 2
    prob2, keep2 = P.make_problem(w, warmup=WARMUP_SAMPLES, prune=other_mode, seed=0,
                                  frontier_cap=args.frontier_cap)
    P.poseidon_search(prob2)
    o_ms, o_ev, o_ok = [], 0, True
    for _ in range(max(3, min(100, args.steps // 2))):
        ms_, plan2, st2 = timed_search_call(prob2)
        o_ms.append(ms_)
        o_ev += st2["evaluated"]
        o_ok &= plan2["global_index"] == ref["plan"]["global_index"]
    other_prune = {"prune": other, "time_to_plan_s": sum(o_ms) / len(o_ms) / 1e3,
                   "evaluations_per_step": o_ev / len(o_ms),
                   "evals_per_s": o_ev / (sum(o_ms) / 1e3), "matches_oracle": o_ok}
    # config 3 (L=48, S=8, M=64, 4 A + 4 B stages): the exhaustive search
    # (memory cut only, no stage-level prune) against the oracle's plan, and
    # its leaf kernel's INT32 fraction from a profiled run
    w3 = gen.config3()
    ref3 = _json.load(open(os.path.join(ROOT, "tests", "golden", "search_plans.json")))
    ref3 = ref3.get("config3", {}).get("plan", {})
    prob3, keep3 = P.make_problem(w3, warmup=500, prune=0, seed=0,
                                  frontier_cap=args.frontier_cap)
    prob3p, keep3p = P.make_problem(w3, warmup=500, prune=0, seed=0,
                                    frontier_cap=args.frontier_cap, profile=True)
    P.poseidon_search(prob3)
    c3_ms, c3_ok = [], True
    for _ in range(max(3, min(100, args.steps // 2))):
        ms_, plan3, st3 = timed_search_call(prob3)
        c3_ms.append(ms_)
        c3_ok &= plan3["global_index"] == ref3.get("global_index")
    _, st3p = P.poseidon_search(prob3p)
    leaf3 = st3p["evaluated"] - st3p["warmup_evaluated"]
    ops3 = (3 * 2 * w3.S * w3.M_list[0] + 9 * w3.S) * leaf3
    ach3 = ops3 / max(st3p["ms_leaf"] / 1e3, 1e-12) / 1e12
    exhaustive3 = {"workload": "config 3: L=48, h=5120, S=8, M=64, exactly 4 A + 4 B stages",
                   "prune": "none (memory cut only)",
                   "time_to_plan_s": sum(c3_ms) / len(c3_ms) / 1e3,
                   "evaluations_per_step": st3["evaluated"], "T_us": plan3["T"],
                   "matches_oracle": c3_ok,
                   "leaf_kernel": {"ms": round(st3p["ms_leaf"], 4),
                                   "launches": st3p["leaf_launches"], "bound": "alu",
                                   "achieved": round(ach3, 3), "unit": "Tops/s",
                                   "frac": round(ach3 / peak_alu, 4)}}
    cpu_rate, cpu_n, cpu_t = oracle_sample_rate(args.cpu_seconds)
    # the oracle's time to the plan on this host: configs 1-3 on one core,
    # config 4 on every core (slices dealt round-robin), beside the GPU's
    cpu_ttp = None
    if args.cpu_time_to_plan:
        procs = max(1, os.cpu_count() or 1)
        gpu_plans = {4: (plans[-1]["T"], plans[-1]["global_index"], t_dev / args.steps / 1e3)}
        gpu_plans[3] = (plan3["T"], plan3["global_index"], sum(c3_ms) / len(c3_ms) / 1e3)
        cpu_ttp = oracle_time_to_plan([(1, 1), (2, 1), (3, 1), (4, procs)])
        for e in cpu_ttp:
            ref_c = _json.load(open(os.path.join(ROOT, "tests", "golden",
                                                 "search_plans.json")))[f"config{e['config']}"]
            e["matches_stored_oracle_plan"] = (e["T_us"] == ref_c["plan"]["T"] and
                                               e["global_index"] == ref_c["plan"]["global_index"])
            if e["config"] in gpu_plans:
                T, gi, sec = gpu_plans[e["config"]]
                e["gpu_time_to_plan_s"] = sec
                e["gpu_prune"] = PRUNE_NAMES[args.prune] if e["config"] == 4 else "none"
                e["same_plan_as_gpu"] = e["T_us"] == T and e["global_index"] == gi
        c5_rate, c5_t = oracle_config5_rate(int(args.cpu_config5), procs)
        cpu_ttp.append({"config": 5, "evals_per_s": c5_rate, "processes": procs,
                        "sample": f"first {int(args.cpu_config5)} config-5 candidates",
                        "seconds": round(c5_t, 3)})
    cpu_all = None
    if args.cpu_seconds >= 1.0:
        rate_all, procs, n_all = oracle_all_cores_rate(min(5.0, args.cpu_seconds))
        cpu_all = {"value": rate_all, "unit": "evals/s", "cores": procs, "kind": "oracle",
                   "sample": f"{n_all} config-4 plan evaluations, one single-threaded oracle "
                             f"process per host core, {min(5.0, args.cpu_seconds):.0f} s each"}
    line = {
        "metric": METRIC, "value": value, "unit": "evals/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": t_dev / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int32",
        "data": "synthetic",
        "config": {"workload": WORKLOAD, "warmup_samples": WARMUP_SAMPLES,
                   "prune": PRUNE_NAMES[args.prune], "l2": "flushed (256 MB write) between steps",
                   "parallelism": "replicas" if world > 1 else "single GPU"},
        "value_note": ("evaluations per second of search: every plan whose makespan the "
                       "search computed (the searched plans, the warm-up samples and the "
                       "greedy seeds, see evaluations_per_step) over the device time"),
        "time_to_plan_s": t_dev / args.steps / 1e3,
        "relaxations_per_s": agg["relaxations"] * world / (t_dev / 1e3),
        "evaluations_per_step": agg["evaluated"] / args.steps,
        "frontier_entries_per_step": agg["prefixes"] / args.steps,
        "plan": {"T_us": plans[-1]["T"], "global_index": plans[-1]["global_index"],
                 "tp": plans[-1]["tp"], "D": plans[-1]["D"], "layers": plans[-1]["layers"],
                 "types": plans[-1]["types"], "matches_oracle": parity},
        "kernels": per_kind,
        "kernel_timing": (f"{args.steps} further searches of the same workload with CUDA events "
                          f"around every launch (profile=1): {sum(prof_ms) / len(prof_ms):.3f} "
                          "ms per search"),
        "host_ms_per_step": {k: round(agg[k] / args.steps, 3)
                             for k in ("ms_setup", "ms_warmup", "ms_search")},
        "roofline": roof,
        "int32_probe": probe,
        "other_prune": other_prune,
        "eval_throughput": evals,
        "eval_sweep": sweep,
        "eval_throughput_eager": evals_eager,
        "eval_throughput_interleaved": evals_il,
        "eval_throughput_config3": evals_c3,
        "eager_search": eager_search,
        "config3_exhaustive": exhaustive3,
        "ridge_search": ridge_lines,
        "per_stage_tp_search": per_stage_tp,
        "interleaved_search": il_lines,
        "cpu_baseline": {"value": cpu_rate, "unit": "evals/s", "cores": 1, "kind": "oracle",
                         "sample": f"{cpu_n} config-4 plan evaluations (S=8, M=32, L=80) in "
                                   f"{cpu_t:.1f} s, single-threaded oracle"},
        "cpu_baseline_all_cores": cpu_all,
        "cpu_time_to_plan": cpu_ttp,
        "e2e": {"value": e2e, "unit": "evals/s", "h2d_bytes_per_step": int(tab_bytes),
                "d2h_bytes_per_step": int(P.binding.C.sizeof(P.binding.pos_plan))},
        "gpu_launches": int(agg["launches"]),
        "clocks": clk,
    }
    print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    # 1500 config-4 searches (~1 s) so that the clock sampler sees the timed region
    ap.add_argument("--steps", type=int, default=1500)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--cpu-time-to-plan", type=int, choices=[0, 1], default=1,
                    help="time the oracle's search on configs 1-4 on this host's cores")
    ap.add_argument("--cpu-config5", type=float, default=1e6,
                    help="config-5 candidates the oracle evaluates on all cores")
    ap.add_argument("--backend", choices=["nccl", "gloo"], default="nccl")
    ap.add_argument("--eval-sizes", type=float, nargs="*", default=[1e7],
                    help="config-5 batch sizes for the evaluator measurement")
    ap.add_argument("--eval-sweep", type=float, nargs="*", default=[1e4, 1e5, 1e6, 1e8],
                    help="further config-5 batch sizes (1F1B), reported as eval_sweep")
    ap.add_argument("--prune", type=int, choices=[1, 2], default=2,
                    help="stage-level prune: 1 = Eq. 2 as printed, 2 = tightened bound")
    ap.add_argument("--frontier-cap", type=int, default=0,
                    help="frontier entries per depth (0 = library default)")
    ap.add_argument("--eval-only", type=int, choices=[0, 1, 2], default=None,
                    help="only the evaluator measurement, under this schedule (0 = 1F1B, "
                         "1 = Eager 1F1B, 2 = Interleaved 1F1B), --steps calls per batch "
                         "size, one JSON line per size (for profiling)")
    args = ap.parse_args()
    rank, world, local_rank = dist_env()
    if args.eval_only is not None:
        import torch
        import paper_2609_06086_gb300 as P
        peak = torch.cuda.get_device_properties(0).multi_processor_count * SM_LANES * 2070e6 / 1e12
        for n in args.eval_sizes:
            print(json.dumps(eval_throughput(P, torch, int(n), args.steps, peak,
                                             schedule=args.eval_only)), flush=True)
        return
    if args.impl == "reference":
        run_reference(args, rank, world)
    else:
        run_ours(args, rank, world, local_rank)


if __name__ == "__main__":
    main()
