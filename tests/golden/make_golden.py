"""Write ``config_results.json``: oracle results for the five standard workloads.

Calls only the CPU oracle (``oracle/``) and the input generator.  Run from the
repository root:  python tests/golden/make_golden.py [--threads T]
Takes minutes: the N=19 workload is 3^19 = 1,162,261,467 simulated mappings.
"""
import argparse
import json
import os
import sys
import time

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from paper_2607_22242_gb300 import scenarios as S  # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "config_results.json")


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--threads", type=int, default=oracle.default_threads())
    args = ap.parse_args()
    res = {"_about": "Oracle results for the standard workloads (scenarios.config(i)); written by "
                     "tests/golden/make_golden.py from the CPU oracle only. 'summary' covers every "
                     "mapping: feasible count, sum of feasible makespans, order-sensitive hash "
                     "(sum of makespan*(idx*2654435761+1) mod 2^64, infeasible = 0xFFFFFFFF) and the argmin.",
           "configs": {}}
    for i in range(4):
        scn = S.config(i)
        t = time.time()
        summ = oracle.summary_range(scn, 0, 3 ** scn.n, args.threads)
        res["configs"][str(i)] = dict(name=S.CONFIG_NAMES[i], sha256=S.sha256_of([scn]), n=scn.n,
                                      mappings=3 ** scn.n, summary=summ)
        print(f"config {i}: {summ} ({time.time() - t:.1f}s, {args.threads} threads)", flush=True)
    batch = S.config4()
    t = time.time()
    idx, ms = oracle.search_batch(batch, args.threads)
    res["configs"]["4"] = dict(name=S.CONFIG_NAMES[4], sha256=S.sha256_of(batch), n=10, count=len(batch),
                               mappings=len(batch) * 3 ** 10,
                               best_index=[int(v) for v in idx], best_makespan=[int(v) for v in ms])
    print(f"config 4: {len(batch)} scenarios ({time.time() - t:.1f}s)", flush=True)
    with open(OUT, "w") as fh:
        json.dump(res, fh, indent=1)


if __name__ == "__main__":
    main()
