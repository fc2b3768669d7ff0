"""Plant plausible slips in a copy of the oracle (on the CPU) and check that the pins catch each one.

Every mutant is a one-token edit of ``oracle/bf_oracle.cpp`` compiled to a
temporary library; the real source is never touched.
"""
import os

import pytest

import oracle
import pins

MUTANTS = {
    "ceil->floor at GPU completion": ("t_gpu = T + ceil_div((v_min - V) * s.slowdown[running_gpu], 1ull << 20);",
                                       "t_gpu = T + ((v_min - V) * s.slowdown[running_gpu] >> 20);"),
    "slowdown index k-1": ("s.slowdown[running_gpu], 1ull << 20", "s.slowdown[running_gpu - 1 > 0 ? running_gpu - 1 : 1], 1ull << 20"),
    "no V advance at CPU events": ("if (running_gpu > 0) V += ((t_cpu - T) << 20) / s.slowdown[running_gpu];", ""),
    "transfer dropped from gpu_now": ("start_on_gpu(v, s.gpu[v] + s.xfer[v]);", "start_on_gpu(v, s.gpu[v]);"),
    "load dropped from gpu_queue": ("start_on_gpu(head, s.load[head] + s.gpu[head] + s.xfer[head]);",
                                    "start_on_gpu(head, s.gpu[head] + s.xfer[head]);"),
    "queue bypass allowed": ("if (head < 0 || ready_time[v] < ready_time[head]) head = v;",
                             "if (live_vram + s.vram[v] <= s.budget && (head < 0 || ready_time[v] < ready_time[head])) head = v;"),
    "queue ties to higher index": ("ready_time[v] < ready_time[head]) head = v;", "ready_time[v] <= ready_time[head]) head = v;"),
    "VRAM not released": ("live_vram -= s.vram[v];", ""),
    "queue never freed": ("if (mode[v] == kGpuQueue) queue_busy = false;", ""),
    "strict budget test for gpu_now": ("if (live_vram > s.budget) {", "if (live_vram >= s.budget) {"),
    "queued tool ignores budget": ("if (!queue_busy && live_vram + s.vram[head] <= s.budget) {", "if (!queue_busy) {"),
    "CPU tool pays transfer": ("cpu_end[v] = T + s.cpu[v];", "cpu_end[v] = T + s.cpu[v] + s.xfer[v];"),
    "digits reversed": ("mode[i] = (int)(idx % 3);", "mode[n - 1 - i] = (int)(idx % 3);"),
    "argmin ties to higher index": ("(ms == makespan && idx < index)", "(ms == makespan && idx > index)"),
    "GPU tools not slowed by contention": ("(v_min - V) * s.slowdown[running_gpu]", "(v_min - V) * 1024"),
    "binary member indexed in base 2": ("for (int i = 0; i < n; ++i, p *= 3)\n    if ((b >> i) & 1) idx += p;",
                                        "for (int i = 0; i < n; ++i, p *= 2)\n    if ((b >> i) & 1) idx += p;"),
    "binary member skips the top tool": ("for (int i = 0; i < n; ++i, p *= 3)\n    if ((b >> i) & 1) idx += p;",
                                         "for (int i = 0; i + 1 < n; ++i, p *= 3)\n    if ((b >> i) & 1) idx += p;"),
    "edges out of tool 30 ignored": ("if (((s.pred[v] >> u) & 1u) && status[u] != kDone) return false;",
                                     "if (u != 30 && ((s.pred[v] >> u) & 1u) && status[u] != kDone) return false;"),
    "batch record indexed from the thread's first": ("unpack(flats + j * kFlatWords)", "unpack(flats + (j - lo) * kFlatWords)"),
    "summary hash multiplier mistyped": ("hash[t] += ms * (idx * 2654435761ull + 1);",
                                         "hash[t] += ms * (idx * 2654435769ull + 1);"),
    "summary counts infeasible mappings": ("        if (ms != kInfeasibleMakespan) {\n          feasible[t] += 1;",
                                           "        if (true) {\n          feasible[t] += 1;"),
    "summary keeps one thread's sum": ("out[1] += total[t];", "out[1] = total[t];"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, tmp_path):
    before, after = MUTANTS[name]
    src = open(oracle.SOURCE).read()
    assert src.count(before) == 1, f"mutation anchor not found once: {before!r}"
    mutant_src = tmp_path / "mutant.cpp"
    mutant_src.write_text(src.replace(before, after))
    lib = oracle.OracleLib(oracle.build(force=True, source=str(mutant_src), out=str(tmp_path / "libmutant.so")))
    caught = []
    for check in pins.ALL_CHECKS:
        try:
            check(lib)
        except AssertionError:
            caught.append(check.__name__)
    assert caught, f"no pin caught mutant: {name}"
