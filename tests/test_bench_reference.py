"""The bench's reference arm (the CPU oracle timed on host cores) prints one JSON line with
the contract's keys; it needs no GPU (runs here on the tiny configuration)."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_the_contract_line():
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--config", "tiny",
                        "--steps", "2", "--warmup", "1"], cwd=ROOT, capture_output=True, text=True,
                       timeout=600, env={**os.environ, "CUDA_VISIBLE_DEVICES": ""})
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "config", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["steps"] == 2 and d["warmup"] == 1 and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0


def _bench():
    import importlib.util
    spec = importlib.util.spec_from_file_location("bench_mod", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_timed_plan_times_exactly_k_steps_spread_over_the_horizon():
    """The bench times exactly K steps: K // T whole trajectories, then K % T positions, one
    at the midpoints of K % T equal slices of the horizon (so a short run samples all of it)."""
    plan_of = _bench().timed_plan
    for T in (1, 6, 10, 30, 50, 64):
        for K in (1, 3, T - 1, T, T + 1, 2 * T + 5, 20):
            if K < 1:
                continue
            plan = plan_of(K, T)
            assert sum(len(p) for p in plan) == K
            for traj in plan:
                assert traj == sorted(set(traj)) and 1 <= traj[0] and traj[-1] <= T
            full, rem = divmod(K, T)
            assert all(p == list(range(1, T + 1)) for p in plan[:full])
            if rem:
                last = plan[-1]
                for i, s in enumerate(last):  # step s holds the midpoint of slice i
                    assert s - 1 <= (i + 0.5) * T / rem < s
    assert plan_of(20, 64) == [[2, 5, 9, 12, 15, 18, 21, 25, 28, 31, 34, 37, 41, 44, 47, 50, 53, 57, 60, 63]]
