"""Write tests/golden/search_plans.json: the oracle's exact search result for
the four search workloads (configs 1-4 of gen/), under 1F1B ("configN") and
Eager 1F1B ("configN_eager"), so GPU tests and the bench can compare against
the oracle without re-running its slowest search (config 4 takes minutes
single-threaded).  Calls only oracle/ and gen/.

    python tests/golden/make_search_plans.py [--configs 1 2 3 4] [--schedules 0 1] [--ridge]

With --ridge the searches use the layer-level (ridge) rule of Theorem 2 and
are stored as "configN_ridge" / "configN_eager_ridge".  With
--interleaved V [V ...] the oracle's Interleaved 1F1B search (V chunks per
device over the config's S devices) is stored as "configN_il_vV" instead.
With --per-stage-tp the search over config 4's tables with a TP degree per
stage (gen.config4_per_stage_tp, POS_PLACE_DEVICES) is stored as
"config4_per_stage_tp" instead.
"""
import argparse
import json
import os
import sys
import time

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import gen  # noqa: E402
import oracle  # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "search_plans.json")


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--configs", type=int, nargs="*", default=[1, 2, 3, 4])
    ap.add_argument("--schedules", type=int, nargs="*", default=[0, 1],
                    help="0 = 1F1B, 1 = Eager 1F1B")
    ap.add_argument("--ridge", action="store_true", help="layer-level (ridge) pruning")
    ap.add_argument("--interleaved", type=int, nargs="*", default=None,
                    help="V values: Interleaved 1F1B searches instead")
    ap.add_argument("--per-stage-tp", action="store_true",
                    help="config 4 with a TP degree per stage instead")
    args = ap.parse_args()
    data = json.load(open(OUT)) if os.path.exists(OUT) else {}
    if args.per_stage_tp:
        w = gen.config4_per_stage_tp()
        t0 = time.time()
        plan, stats = oracle.search(w, prune=True, warmup=500, seed=0)
        data["config4_per_stage_tp"] = dict(workload=w.name, seed=w.seed, schedule=0,
                                            plan=plan, oracle_stats=stats,
                                            oracle_seconds=round(time.time() - t0, 2))
        print("config4_per_stage_tp", plan, flush=True)
        with open(OUT, "w") as f:
            json.dump(data, f, indent=1, sort_keys=True)
        return
    if args.interleaved:
        for c in args.configs:
            for V in args.interleaved:
                w = gen.get_config(c)
                t0 = time.time()
                plan, stats = oracle.search_interleaved(w, V, prune=True)
                key = f"config{c}_il_v{V}"
                data[key] = dict(workload=w.name, seed=w.seed, schedule=2, V=V, plan=plan,
                                 oracle_stats=stats, oracle_seconds=round(time.time() - t0, 2))
                print(key, plan, flush=True)
                with open(OUT, "w") as f:
                    json.dump(data, f, indent=1, sort_keys=True)
        return
    for sched in args.schedules:
        for c in args.configs:
            w = gen.get_config(c)
            t0 = time.time()
            plan, stats = oracle.search(w, prune=True, warmup=500, seed=0, schedule=sched,
                                        ridge=args.ridge)
            key = f"config{c}" + ("_eager" if sched == 1 else "") + ("_ridge" if args.ridge else "")
            data[key] = dict(workload=w.name, seed=w.seed, schedule=sched, ridge=args.ridge,
                             plan=plan,
                             oracle_stats=stats, oracle_seconds=round(time.time() - t0, 2))
            print(key, plan, flush=True)
    with open(OUT, "w") as f:
        json.dump(data, f, indent=1, sort_keys=True)


if __name__ == "__main__":
    main()
