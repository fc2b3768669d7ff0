"""Run one kernel of the search on a chosen range, for timing and profiling.

  python -m paper_2607_22242_gb300.profile_case --kernel search --config 3 --count 67108864 --reps 3
  python -m paper_2607_22242_gb300.profile_case --kernel eval --config 2 --count 16777216
  python -m paper_2607_22242_gb300.profile_case --kernel batch --batch 1024
  python -m paper_2607_22242_gb300.profile_case --kernel list --config 3 --count 16777216
  python -m paper_2607_22242_gb300.profile_case --kernel whatif --config 3 --reps 20
  python -m paper_2607_22242_gb300.profile_case --kernel tree --workload wide32 --space 3

Prints one line per repetition (CUDA-event time of the call and mappings/s).
Sized so that a profiler capture of one launch stays short.
"""
from __future__ import annotations

import argparse
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--kernel", choices=("search", "pruned", "eval", "batch", "list", "whatif", "tree"),
                    default="search")
    ap.add_argument("--config", type=int, default=3)
    ap.add_argument("--workload", default=None, help="wide28 | wide32 | layered24 (instead of --config)")
    ap.add_argument("--space", type=int, default=3, help="tree search: 3 = full space, 2 = binary")
    ap.add_argument("--no-prune", action="store_true", help="tree search: simulate every mapping")
    ap.add_argument("--first", type=int, default=0)
    ap.add_argument("--count", type=int, default=1 << 26)
    ap.add_argument("--batch", type=int, default=1024, help="scenarios for --kernel batch (config 4 prefix)")
    ap.add_argument("--reps", type=int, default=3)
    args = ap.parse_args()

    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_22242_gb300 import bf
    from paper_2607_22242_gb300 import scenarios as S

    torch.cuda.set_device(0)
    stream = torch.cuda.current_stream()
    if args.kernel == "batch":
        batch = S.config4(args.batch)
        work = len(batch) * 3 ** 10
        packed = bf.pack_descs(batch)  # the C caller's desc array, packed once
        call = lambda: bf.search_batch(batch, stream, packed)
    else:
        scn = getattr(S, args.workload)() if args.workload else S.config(args.config)
        count = min(args.count, 3 ** scn.n - args.first)
        work = count
        h = bf.create_scenario(scn)
        if args.kernel == "tree":  # branch and bound over the chosen space (count ignored)
            work = args.space ** scn.n
            stats = {}

            def call():
                res, st = bf.search_tree(h, args.space, not args.no_prune, None, stream)
                stats.update(st)
                return res
        elif args.kernel == "search":
            call = lambda: bf.search_range(h, args.first, count, stream)
        elif args.kernel == "pruned":  # branch and bound over the whole space (count ignored)
            work = 3 ** scn.n
            call = lambda: bf.search_pruned(h, None, stream)
        elif args.kernel == "list":  # uniformly random mapping indices of the whole space
            g = torch.Generator(device="cuda").manual_seed(1)
            idx = torch.randint(0, 3 ** scn.n, (count,), device="cuda", generator=g, dtype=torch.int64)
            ms = torch.empty(count, dtype=torch.int32, device="cuda")
            fe = torch.empty(count, dtype=torch.uint8, device="cuda")
            call = lambda: bf.eval_indices(h, idx, ms, fe, stream)
        elif args.kernel == "whatif":  # around the optimum of the scenario
            base = bf.search_best(h, stream).index
            work = len(bf.whatif(h, base, stream))
            call = lambda: bf.whatif(h, base, stream)
        else:
            ms = torch.empty(count, dtype=torch.int32, device="cuda")
            fe = torch.empty(count, dtype=torch.uint8, device="cuda")
            call = lambda: bf.eval_mappings(h, args.first, count, ms, fe, stream)
    for rep in range(args.reps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        out = call()
        b.record(stream)
        b.synchronize()
        t = a.elapsed_time(b)
        print(f"{args.kernel} rep {rep}: {t:.3f} ms, {work / (t / 1e3):.4g} mappings/s"
              + (f", best {out.index}/{out.makespan_us}" if args.kernel in ("search", "pruned", "tree") else "")
              + (f", {stats}" if args.kernel == "tree" else ""), flush=True)


if __name__ == "__main__":
    main()
