"""bench.py's reference arm prints the JSON line the measurement contract asks for
(the oracle timed on the host cores, on the tiny workload so that it takes seconds)."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def test_reference_arm_json_line():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--config", "1",
                          "--steps", "2", "--warmup", "1"], capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, out.stdout
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
                "vs_baseline", "dtype", "data", "config", "impl", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["impl"] == "reference" and d["steps"] == 2 and d["warmup"] == 1
    assert d["value"] > 0 and d["higher_is_better"] is True and d["config"]["workload"].startswith("tiny")
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1 and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_trace_schedule_of_the_long_trace():
    """The long-trace mode compresses whenever the cache reaches L rows: after a 128-token prompt and
    32768 decode steps that is once at step 4095 (128 + 4096 = 4224 rows) and then every 128 steps,
    225 compresses in all."""
    import bench
    from paper_2609_04971_gb300.workloads import QWEN3_8B_TRACE as T
    sched = bench.trace_schedule(T.prefill, T.budget, T.L - T.budget, T.trace_steps)
    assert len(sched) == 225 and sched[0] == T.L - T.prefill - 1
    assert all(b - a == T.L - T.budget for a, b in zip(sched, sched[1:]))
    assert bench.trace_schedule(10, 8, 4, 1) == [] and bench.trace_schedule(10, 8, 4, 6) == [1, 5]


def test_trace_phases_follow_algorithm_2():
    """Algorithm 2: a decode step feeds the observation buffer while the cache (after its token) holds at
    most B_max - n_recent rows, keeps its query as a recent one while it holds more, and the step that
    reaches B_max evicts to B_min.  Here B_min = 8, B_max = 12, n_recent = 2, a 5-row prompt."""
    import bench
    ph = bench.trace_phases(prefill=5, b_min=8, b_max=12, window=2, steps=14)
    # L after each step: 6..12 (evict), 9, 10, 11, 12 (evict), 9, 10, 11
    assert ph == ["obs"] * 5 + ["recent"] * 2 + ["obs"] * 2 + ["recent"] * 2 + ["obs"] * 2 + ["recent"]
    sched = bench.trace_schedule(5, 8, 4, 14)
    assert sched == [6, 10]
    # every eviction is preceded by exactly n_recent recent-phase steps
    for s in sched:
        assert ph[s - 1:s + 1] == ["recent", "recent"] and ph[s - 2] == "obs"
    # the paper's 7/8 ratio on the long trace: B_min 4096 -> B_max 4681, n_recent 8
    ph = bench.trace_phases(128, 4096, 4681, 8, 32768)
    sched = bench.trace_schedule(128, 4096, 4681 - 4096, 32768)
    assert all(ph[s] == "recent" and ph[s - 7] == "recent" and ph[s - 8] == "obs" for s in sched)
    assert sum(p == "recent" for p in ph) >= 8 * len(sched)
