"""Pins for the CPU oracle: checks against facts that do not come from the oracle.

Each ``check_*`` takes an :class:`oracle.OracleLib` and raises AssertionError on
a mismatch.  They are run on the real oracle (``test_oracle_pins.py``) and on
deliberately broken copies of it (``test_oracle_mutants.py``) to show that a
plausible slip in the oracle fails at least one of them.

Sources of truth:
* hand-worked examples (``golden/hand_examples.json``), worked out from the
  model's rules (§2.1, Factor A/B of §2.3, Table 1 caption);
* closed forms: serial chains, identical fan-outs, the all-cpu critical path;
* a textbook special case: with no contention, no gpu_queue and no VRAM
  pressure every makespan is the longest path of the DAG under per-mode
  durations (critical-path DP);
* invariants: the argmin is feasible and no worse than all-cpu; a fan-out from
  t=0 is infeasible exactly when its gpu_now footprints exceed M; contention
  never shortens a feasible mapping without gpu_queue;
* the paper's printed numbers: Table 1 speedups (gpu_now = GPU time, queued =
  GPU + Load), Table 3 totals and feasibility (§4.4, §4.5), Figure 7's
  per-probe memory and status;
* a structurally different Python restatement (``oracle.pysim``) on every
  mapping of small random DAGs, and the exact rational model
  (``oracle.exact``) within its rounding bound.
"""
from __future__ import annotations

import json
import math
import os

import numpy as np

from paper_2607_22242_gb300 import scenarios as S
from paper_2607_22242_gb300.scenarios import CPU, GPU_NOW, GPU_QUEUE, Scenario

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
INF = 0xFFFFFFFF
MODE_OF = {"cpu": CPU, "gpu_now": GPU_NOW, "gpu_queue": GPU_QUEUE}


def _load(name):
    with open(os.path.join(GOLDEN, name)) as fh:
        return json.load(fh)


def _chain(n, c, g, x, l, m, budget, f):
    return Scenario(n, [0] + [1 << (i - 1) for i in range(1, n)], c, g, x, l, m, budget, f)


def _longest_path(scn, dur):
    """Critical-path length: finish[v] = dur[v] + max(finish[u] for u in pred(v))."""
    finish = []
    for v in range(scn.n):
        start = max([finish[u] for u in range(v) if (scn.pred_mask[v] >> u) & 1], default=0)
        finish.append(start + dur[v])
    return max(finish)


# ---------------------------------------------------------------------------

def check_hand_examples(lib):
    for ex in _load("hand_examples.json")["examples"]:
        scn = Scenario.from_dict(ex["scenario"])
        for idx, want in ex["expected"].items():
            got = lib.evaluate(scn, int(idx))
            assert got == want, f"{ex['name']}: idx {idx}: {got} != {want}"
        if "argmin" in ex:
            assert list(lib.search(scn)) == ex["argmin"], ex["name"]


def check_chain_closed_forms(lib, trials=40, seed=11):
    rng = np.random.default_rng(seed)
    for _ in range(trials):
        n = int(rng.integers(1, 9))
        c = [int(v) for v in rng.integers(1, 100000, n)]
        g = [int(v) for v in rng.integers(1, 100000, n)]
        x = [int(v) for v in rng.integers(0, 30000, n)]
        l = [int(v) for v in rng.integers(0, 50000, n)]
        m = [int(v) for v in rng.integers(1, 5000, n)]
        f = S.random_small(rng, 2).slowdown_q10  # any table: a chain never runs two GPU tools
        scn = _chain(n, c, g, x, l, m, max(m), f)
        all_now = sum(3 ** i for i in range(n))
        assert lib.evaluate(scn, 0) == sum(c)
        assert lib.evaluate(scn, all_now) == sum(g) + sum(x)
        assert lib.evaluate(scn, 2 * all_now) == sum(l) + sum(g) + sum(x)
        # any mixed mapping of a chain: the sum of per-mode durations
        for idx in rng.integers(0, 3 ** n, 8):
            modes = S.mapping_modes(int(idx), n)
            dur = [(c[i], g[i] + x[i], l[i] + g[i] + x[i])[a] for i, a in enumerate(modes)]
            assert lib.evaluate(scn, int(idx)) == sum(dur)
        # a tool larger than the budget: gpu_now or gpu_queue on it is infeasible
        big = Scenario(n, scn.pred_mask, c, g, x, l, [max(m) + 1] + m[1:], max(m), f)
        assert lib.evaluate(big, 1) == INF and lib.evaluate(big, 2) == INF


def check_identical_fanout(lib, seed=12):
    rng = np.random.default_rng(seed)
    for n in range(1, 13):
        w = int(rng.integers(1, 200000))
        f = S.slowdown_linear(int(rng.integers(0, 80)))
        scn = Scenario(n, [0] * n, [10 ** 7] * n, [w] * n, [0] * n, [0] * n, [1] * n, n, f)
        all_now = sum(3 ** i for i in range(n))
        want = -(-w * f[n] // 1024)  # ceil(w * f[n] / 1024)
        assert lib.evaluate(scn, all_now) == want, (n, w, f[n])


def check_longest_path(lib, trials=30, seed=13):
    """No contention, no queue, no VRAM pressure: every makespan is a critical path."""
    rng = np.random.default_rng(seed)
    for _ in range(trials):
        n = int(rng.integers(1, 8))
        scn = S.random_small(rng, n, tight=False, contention=False, max_time=1000)
        ms, fe = lib.eval_range(scn, 0, 3 ** n)
        for idx in range(3 ** n):
            modes = S.mapping_modes(idx, n)
            if GPU_QUEUE in modes:
                continue
            dur = [scn.cpu_us[i] if a == CPU else scn.gpu_us[i] + scn.xfer_us[i] for i, a in enumerate(modes)]
            assert fe[idx] == 1 and int(ms[idx]) == _longest_path(scn, dur), (scn, idx)


def check_all_cpu_is_critical_path(lib, trials=40, seed=14):
    rng = np.random.default_rng(seed)
    for _ in range(trials):
        n = int(rng.integers(1, 12))
        scn = S.random_small(rng, n, tight=True, max_time=500)
        assert lib.evaluate(scn, 0) == _longest_path(scn, scn.cpu_us)


def check_argmin_invariants(lib, trials=40, seed=15):
    rng = np.random.default_rng(seed)
    for _ in range(trials):
        n = int(rng.integers(1, 7))
        scn = S.random_small(rng, n)
        ms, fe = lib.eval_range(scn, 0, 3 ** n)
        idx, best = lib.search(scn)
        assert fe[0] == 1 and fe[idx] == 1
        assert best == int(ms[idx]) <= int(ms[0])
        feas = np.flatnonzero(fe)
        assert best == int(ms[feas].min())
        assert idx == int(feas[np.argmax(ms[feas] == best)])  # lowest index among ties
        assert np.all(ms[fe == 0] == INF)


def check_fanout_feasibility(lib, trials=40, seed=16):
    """Fan-out from t=0 with every footprint <= M: infeasible iff sum(gpu_now m) > M."""
    rng = np.random.default_rng(seed)
    for _ in range(trials):
        n = int(rng.integers(1, 7))
        base = S.random_small(rng, n, edge_p=0.0)
        budget = int(rng.integers(max(base.vram_mib), 3 * max(base.vram_mib) + 1))
        scn = Scenario(n, [0] * n, base.cpu_us, base.gpu_us, base.xfer_us, base.load_us,
                       base.vram_mib, budget, base.slowdown_q10)
        ms, fe = lib.eval_range(scn, 0, 3 ** n)
        for idx in range(3 ** n):
            modes = S.mapping_modes(idx, n)
            now_mem = sum(scn.vram_mib[i] for i, a in enumerate(modes) if a == GPU_NOW)
            assert bool(fe[idx]) == (now_mem <= budget), (scn, idx)


def check_contention_monotone(lib, trials=40, seed=17):
    """Without gpu_queue, a mapping feasible with and without contention is never faster with it."""
    rng = np.random.default_rng(seed)
    for _ in range(trials):
        n = int(rng.integers(1, 7))
        scn = S.random_small(rng, n, max_time=int(rng.choice([20, 500])))
        flat = Scenario(**{**scn.to_dict(), "slowdown_q10": S.slowdown_flat()})
        ms_f, fe_f = lib.eval_range(scn, 0, 3 ** n)
        ms_1, fe_1 = lib.eval_range(flat, 0, 3 ** n)
        for idx in range(3 ** n):
            if GPU_QUEUE in S.mapping_modes(idx, n) or not (fe_f[idx] and fe_1[idx]):
                continue
            assert ms_f[idx] >= ms_1[idx], (scn, idx)


def check_against_pysim(lib, trials=120, seed=18):
    from oracle import pysim
    rng = np.random.default_rng(seed)
    for t in range(trials):
        n = int(rng.integers(1, 6 if t % 4 else 7))
        scn = S.random_small(rng, n, edge_p=float(rng.choice([0.0, 0.3, 0.7])),
                             tight=bool(t % 3), contention=bool(t % 5),
                             max_time=int(rng.choice([6, 30, 2000])))
        ms, fe = lib.eval_range(scn, 0, 3 ** n)
        for idx in range(3 ** n):
            want, ok = pysim.evaluate(scn, idx)
            assert (int(ms[idx]), bool(fe[idx])) == (want if ok else INF, ok), (scn, idx)


def check_rational_bound(lib, trials=60, seed=19):
    """Mappings without gpu_queue whose feasibility agrees: |integer - exact| <= 2N*ceil(f[N]/1024)."""
    from oracle import exact
    rng = np.random.default_rng(seed)
    for _ in range(trials):
        n = int(rng.integers(1, 6))
        scn = S.random_small(rng, n, max_time=int(rng.choice([10, 1000])))
        ms, fe = lib.eval_range(scn, 0, 3 ** n)
        bound = 2 * n * math.ceil(scn.slowdown_q10[n] / 1024)
        for idx in range(3 ** n):
            modes = S.mapping_modes(idx, n)
            if GPU_QUEUE in modes:
                continue
            t, ok, _ = exact.simulate(scn, modes)
            if ok != bool(fe[idx]) or not ok:
                continue
            assert abs(int(ms[idx]) - t) <= bound, (scn, idx, int(ms[idx]), float(t))


# ---------------------------------------------------------------------------
# The paper's printed numbers.
# ---------------------------------------------------------------------------

def _one_tool(cpu_ms, gpu_ms, load_ms, vram):
    us = lambda v: int(round(v * 1000))
    return Scenario(1, [0], [us(cpu_ms)], [us(gpu_ms)], [0], [us(load_ms)], [vram], vram, S.slowdown_flat())


def _printed_close(value, printed):
    if printed.startswith("<"):
        return value < float(printed[1:])
    decimals = len(printed.split(".")[1]) if "." in printed else 0
    return abs(value - float(printed)) <= 10.0 ** (-decimals) + 1e-12


def check_table1_speedups(lib):
    """Table 1: CPU/GPU speedup from the cpu and gpu_now runs, CPU/(GPU+Load) from the queued run."""
    for t in _load("paper_table1.json")["tools"]:
        if t["vram_mb"] is None:
            continue
        scn = _one_tool(t["cpu_ms"], t["gpu_ms"], t["load_ms"], t["vram_mb"])
        cpu, now, queued = (lib.evaluate(scn, i) for i in range(3))
        assert _printed_close(cpu / now, t["speedup"]), (t["tool"], cpu / now)
        assert _printed_close(cpu / queued, t["queue_speedup"]), (t["tool"], cpu / queued)


def _fanout(tools, budget):
    n = len(tools)
    us = lambda v: int(round(v * 1000))
    return Scenario(n, [0] * n, [us(t["cpu_ms"]) for t in tools], [us(t["gpu_ms"]) for t in tools],
                    [0] * n, [us(t["load_ms"]) for t in tools], [t["vram_mb"] for t in tools],
                    budget, S.slowdown_linear())


def check_table3_feasibility(lib):
    tools = {t["tool"]: t for t in _load("paper_table1.json")["tools"]}
    t3 = _load("paper_table3.json")
    by_id = {s["id"]: s for s in t3["scenarios"]}
    for case in t3["feasibility"]["cases"]:
        sc = by_id[case["scenario"]]
        scn = _fanout([tools[name] for name in sc["tools"]], sc["budget"])
        idx = S.mapping_index([MODE_OF[m] for m in case["modes"]])
        assert (lib.evaluate(scn, idx) != INF) == case["feasible"], case


def check_fig7_probes(lib):
    """Figure 7: status of every probe; printed memory = gpu_now footprints within 2 MB."""
    f7 = _load("paper_fig7.json")
    tools = [dict(cpu_ms=t["cpu"], gpu_ms=t["gpu"], load_ms=t["load"], vram_mb=t["mem"]) for t in f7["tools"]]
    for p in f7["probes"]:
        idx = S.mapping_index([MODE_OF[m] for m in p["modes"]])
        assert (lib.evaluate(_fanout(tools, f7["budget_mb"]), idx) != INF) == p["feasible"], p
        # the memory the probe holds at once lies in [mem-2, mem+2]
        assert lib.evaluate(_fanout(tools, p["mem"] + 2), idx) != INF, p
        assert lib.evaluate(_fanout(tools, p["mem"] - 3), idx) == INF, p


ALL_CHECKS = [
    check_hand_examples, check_chain_closed_forms, check_identical_fanout, check_longest_path,
    check_all_cpu_is_critical_path, check_argmin_invariants, check_fanout_feasibility,
    check_contention_monotone, check_against_pysim, check_rational_bound,
    check_table1_speedups, check_table3_feasibility, check_fig7_probes,
]


def check_fig7_whatif(lib):
    """Figure 7's what-if block: around the mapping of the monitor's second round (A:GN B:GN C:GQ D:CPU)
    Algorithm 1 reprobes C -> gpu_now, which exceeds 1100 MB, and then swaps C
    with each gpu_now tool; every probe printed there appears with its status
    and, for swaps, the printed full mapping."""
    from oracle import whatif as W
    f7 = _load("paper_fig7.json")
    tools = [dict(cpu_ms=t["cpu"], gpu_ms=t["gpu"], load_ms=t["load"], vram_mb=t["mem"]) for t in f7["tools"]]
    scn = _fanout(tools, f7["budget_mb"])
    base = S.mapping_index([GPU_NOW, GPU_NOW, GPU_QUEUE, CPU])
    probes = W.whatif(scn, base, evaluate=lib.evaluate)
    singles = {(p[1], p[2]): p for p in probes if p[0] == "single"}
    swaps = {(p[1], p[3]): p for p in probes if p[0] == "swap"}
    A, B, C, D = range(4)
    assert len(singles) == 8
    for (tool, mode), feasible in (((A, CPU), True), ((B, CPU), True), ((C, GPU_NOW), False), ((D, GPU_QUEUE), True)):
        assert singles[(tool, mode)][6] == feasible, (tool, mode)
    for (i, j), full in (((C, A), [GPU_QUEUE, GPU_NOW, GPU_NOW, CPU]), ((C, B), [GPU_NOW, GPU_QUEUE, GPU_NOW, CPU])):
        p = swaps[(i, j)]
        assert p[4] == S.mapping_index(full) and p[6], (i, j)
    # Algorithm 1 swaps exactly the blocked tools with each tool on gpu_now.
    blocked = [t for (t, m), p in singles.items() if m == GPU_NOW and not p[6]]
    assert set(swaps) == {(i, j) for i in blocked for j in (A, B)}
    # the swaps follow their single reprobe in the list
    pos = {(p[0], p[1], p[2], p[3]): k for k, p in enumerate(probes)}
    for i, j in swaps:
        assert pos[("swap", i, GPU_NOW, j)] > pos[("single", i, GPU_NOW, None)]


ALL_CHECKS.append(check_fig7_whatif)


# ---------------------------------------------------------------------------
# Scenarios of up to 32 tools, the binary decision space and the segment rule.
# ---------------------------------------------------------------------------

def check_wide_closed_forms(lib, seed=21):
    """Closed forms at 21..32 tools (the last tool sits at bit 31 of every mask)."""
    rng = np.random.default_rng(seed)
    for n in (21, 27, 32):
        c = [int(v) for v in rng.integers(1, 100000, n)]
        g = [int(v) for v in rng.integers(1, 100000, n)]
        x = [int(v) for v in rng.integers(0, 30000, n)]
        l = [int(v) for v in rng.integers(0, 50000, n)]
        m = [int(v) for v in rng.integers(1, 5000, n)]
        scn = _chain(n, c, g, x, l, m, max(m), S.slowdown_linear(35, kmax=n))
        ones = sum(3 ** i for i in range(n))
        assert lib.evaluate(scn, 0) == sum(c)
        assert lib.evaluate(scn, ones) == sum(g) + sum(x)
        assert lib.evaluate(scn, 2 * ones) == sum(l) + sum(g) + sum(x)
        for idx in rng.integers(0, 2 ** 62, 6):
            idx = int(idx) % 3 ** n
            modes = S.mapping_modes(idx, n)
            dur = [(c[i], g[i] + x[i], l[i] + g[i] + x[i])[a] for i, a in enumerate(modes)]
            assert lib.evaluate(scn, idx) == sum(dur), (n, idx)
        # identical fan-out of n tools on gpu_now: each ends at ceil(w f[n] / 1024)
        w = int(rng.integers(1, 200000))
        f = S.slowdown_linear(int(rng.integers(0, 80)), kmax=n)
        fan = Scenario(n, [0] * n, [10 ** 7] * n, [w] * n, [0] * n, [0] * n, [1] * n, n, f)
        assert lib.evaluate(fan, ones) == -(-w * f[n] // 1024), (n, w)
        # one tool over budget, at the top digit
        big = Scenario(n, scn.pred_mask, c, g, x, l, m[:-1] + [max(m) + 1], max(m), scn.slowdown_q10)
        assert lib.evaluate(big, 3 ** (n - 1)) == INF and lib.evaluate(big, 2 * 3 ** (n - 1)) == INF
        # all-cpu mapping of a random DAG: its critical path
        dag = S.random_small(rng, n, tight=True, max_time=500)
        assert lib.evaluate(dag, 0) == _longest_path(dag, dag.cpu_us)


def check_binary_space(lib, trials=40, seed=22):
    """The binary (cpu/gpu_now) optimum: hand-worked values, and every binary mapping of small DAGs."""
    for ex in _load("hand_examples.json")["examples"]:
        scn = Scenario.from_dict(ex["scenario"])
        members = [sum(3 ** i for i in range(scn.n) if (b >> i) & 1) for b in range(2 ** scn.n)]
        if not all(str(i) in ex["expected"] for i in members):
            continue
        feas = [(ex["expected"][str(i)], i) for i in members if ex["expected"][str(i)] != INF]
        want = min(feas)
        assert lib.search_binary(scn) == (want[1], want[0]), ex["name"]
    rng = np.random.default_rng(seed)
    for _ in range(trials):
        n = int(rng.integers(1, 8))
        scn = S.random_small(rng, n)
        ms, fe = lib.eval_range(scn, 0, 3 ** n)
        best = None
        for b in range(2 ** n):
            idx = sum(3 ** i for i in range(n) if (b >> i) & 1)
            if fe[idx] and (best is None or (int(ms[idx]), idx) < best):
                best = (int(ms[idx]), idx)
        assert lib.search_binary(scn) == (best[1], best[0]), scn
        lo = int(rng.integers(0, 2 ** n))
        cnt = int(rng.integers(1, 2 ** n - lo + 1))
        sub = [(int(ms[i]), i) for i in (sum(3 ** k for k in range(n) if (b >> k) & 1) for b in range(lo, lo + cnt))
               if fe[i]]
        got = lib.search_binary_range(scn, lo, cnt)
        assert got == ((min(sub)[1], min(sub)[0]) if sub else (-1, INF)), (scn, lo, cnt)


def check_segments(lib, trials=40, seed=23):
    """Segment rule (oracle.segments): equal to full enumeration, and to the stored
    brute-force optimum of the 19-tool workload."""
    from oracle import segments
    rng = np.random.default_rng(seed)
    for t in range(trials):
        n = int(rng.integers(2, 9))
        scn = S.random_segmented(rng, n, seg_max=int(rng.choice([2, 3, 5])), tight=bool(t % 3),
                                 max_time=int(rng.choice([8, 40, 500])))
        assert segments.bounds(scn)[-1][1] == n
        assert segments.search(scn, lib=lib) == lib.search(scn), scn
        assert segments.search(scn, binary=True, lib=lib) == lib.search_binary(scn), scn
        for idx in rng.integers(0, 3 ** n, 10):
            assert segments.evaluate(scn, int(idx), lib=lib) == lib.evaluate(scn, int(idx)), (scn, idx)
    golden = _load("config_results.json")["configs"]["3"]
    assert segments.search(S.config3(), lib=lib) == (golden["summary"]["best_index"], golden["summary"]["best_makespan"])


def check_degenerate_budgets(lib, trials=30, seed=24):
    """M = 0: every GPU mode is infeasible (gpu_now overflows at start, a queued tool can never fit), so the
    all-cpu mapping is the only feasible one and the optimum is the critical path of CPU times; and a
    budget that fits everything at once with f[k] = 65536 for k >= 2: every mapping stays feasible."""
    rng = np.random.default_rng(seed)
    for _ in range(trials):
        n = int(rng.integers(1, 7))
        base = S.random_small(rng, n, max_time=300)
        zero = Scenario(**{**base.to_dict(), "vram_budget_mib": 0})
        ms, fe = lib.eval_range(zero, 0, 3 ** n)
        assert fe[0] == 1 and not fe[1:].any(), zero
        assert lib.search(zero) == (0, _longest_path(zero, zero.cpu_us))
        steep = Scenario(**{**base.to_dict(), "vram_budget_mib": sum(base.vram_mib),
                            "slowdown_q10": [0, 1024] + [65536] * (len(base.slowdown_q10) - 2)})
        ms, fe = lib.eval_range(steep, 0, 3 ** n)
        assert fe.all(), steep


ALL_CHECKS += [check_wide_closed_forms, check_binary_space, check_segments, check_degenerate_budgets]


# ---------------------------------------------------------------------------
# The aggregating entry points that write the full-size expected values: the
# batch search (per-scenario optima of the 4096-scenario workload) and the
# range summary (feasible count, makespan sum, order-sensitive hash and argmin
# of the 8-, 12-, 16- and 19-tool workloads).  Each is checked against plain
# reductions of the per-mapping makespans, which the pins above fix.
# ---------------------------------------------------------------------------

def _argmin(ms, fe, first=0):
    """(index, makespan) of the lowest feasible makespan, lowest index among ties; (-1, INF) if none."""
    best = None
    for j in range(len(ms)):
        if fe[j] and (best is None or int(ms[j]) < best[1]):
            best = (first + j, int(ms[j]))
    return best if best is not None else (-1, INF)


def check_batch_search(lib, seed=25):
    """Each scenario of a batch gets the argmin of its own 3^n makespans: batches of mixed sizes (1-7
    tools, so consecutive records differ), a one-scenario batch, the last scenario alone, and several
    host threads."""
    rng = np.random.default_rng(seed)
    scns = [S.random_small(rng, int(rng.integers(1, 8)), max_time=int(rng.choice([9, 700])))
            for _ in range(25)]
    want = []
    for s in scns:
        ms, fe = lib.eval_range(s, 0, 3 ** s.n)
        want.append(_argmin(ms, fe))
    for lo, hi, threads in ((0, 25, 1), (0, 25, 4), (0, 1, 1), (24, 25, 1), (7, 19, 3)):
        idx, ms = lib.search_batch(scns[lo:hi], threads)
        got = [(int(i), int(m)) for i, m in zip(idx, ms)]
        assert got == want[lo:hi], (lo, hi, threads)


def check_summary_range(lib, trials=30, seed=26):
    """The range summary equals plain reductions of the range's makespans: the feasible count, the sum of
    feasible makespans, the hash sum_j makespan(j) * (j * 2654435761 + 1) mod 2^64 (infeasible counted
    as 0xFFFFFFFF), summed here in Python integers, and the argmin; on random sub-ranges and over one
    and several host threads."""
    rng = np.random.default_rng(seed)
    for t in range(trials):
        n = int(rng.integers(1, 8))
        scn = S.random_small(rng, n, max_time=int(rng.choice([9, 700])))
        total = 3 ** n
        first = int(rng.integers(0, total)) if t % 3 else 0
        count = int(rng.integers(1, total - first + 1)) if t % 3 else total
        ms, fe = lib.eval_range(scn, first, count)
        got = lib.summary_range(scn, first, count, int(rng.choice([1, 3])))
        feas = [int(m) for m, f in zip(ms, fe) if f]
        assert got["feasible"] == len(feas), (scn, first, count)
        assert got["makespan_sum"] == sum(feas), (scn, first, count)
        h = sum(int(m) * ((first + j) * 2654435761 + 1) for j, m in enumerate(ms)) % (1 << 64)
        assert got["hash"] == h, (scn, first, count)
        best = _argmin(ms, fe, first)
        want = (best[0] if best[0] >= 0 else (1 << 64) - 1, best[1])
        assert (got["best_index"], got["best_makespan"]) == want, (scn, first, count)


ALL_CHECKS += [check_batch_search, check_summary_range]
