"""Write ``wide_results.json``: oracle optima of the workloads beyond 20 tools.

Calls only the CPU oracle (``oracle/``) and the input generator.  Run from the
repository root:  python tests/golden/make_wide_golden.py [--threads T]

* wide28, wide32 (spine + fan-outs, scenarios.wide28/wide32): exact optima of
  the full 3^n space and of the binary cpu/gpu_now space, from the segment
  rule (oracle.segments, pinned against full enumeration).  Seconds.
* layered24: a random layered DAG of 24 tools with no serialisation point;
  the optimum of its binary space by full enumeration of 2^24 mappings.
  Minutes.
"""
import argparse
import json
import os
import sys
import time

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from oracle import segments  # noqa: E402
from paper_2607_22242_gb300 import scenarios as S  # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "wide_results.json")


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--threads", type=int, default=oracle.default_threads())
    args = ap.parse_args()
    res = {"_about": "Oracle optima (index, makespan us) of the workloads beyond 20 tools; written by "
                     "tests/golden/make_wide_golden.py from the CPU oracle only. 'ternary' is the full "
                     "3^n space, 'binary' the cpu/gpu_now space (2^n mappings).",
           "workloads": {}}
    for name in ("wide28", "wide32"):
        scn = getattr(S, name)()
        t = time.time()
        ter = segments.search(scn, threads=args.threads)
        bin_ = segments.search(scn, binary=True, threads=args.threads)
        res["workloads"][name] = dict(name=S.WIDE_NAMES[name], sha256=S.sha256_of([scn]), n=scn.n,
                                      segments=segments.bounds(scn), method="segment rule",
                                      ternary=list(ter), binary=list(bin_))
        print(f"{name}: ternary {ter} binary {bin_} ({time.time() - t:.1f}s)", flush=True)
    scn = S.layered24()
    t = time.time()
    bin_ = oracle.search_binary(scn, args.threads)
    res["workloads"]["layered24"] = dict(name=S.WIDE_NAMES["layered24"], sha256=S.sha256_of([scn]), n=scn.n,
                                         segments=segments.bounds(scn), method="full enumeration",
                                         binary=list(bin_))
    print(f"layered24: binary {bin_} ({time.time() - t:.1f}s, {args.threads} threads)", flush=True)
    with open(OUT, "w") as fh:
        json.dump(res, fh, indent=1)


if __name__ == "__main__":
    main()
