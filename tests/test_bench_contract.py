"""bench.py's output contract on the CPU: the reference arm's JSON line, the warm-up rule,
the per-step statistics and the L2 policy every workload states."""
import json
import os
import subprocess
import sys

import pytest

import bench

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(*args, timeout=300):
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT,
                          env=env, capture_output=True, text=True, timeout=timeout)


def test_reference_arm_prints_one_contract_line():
    r = _run("--impl", "reference", "--steps", "1", "--warmup", "3")
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
                "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["value"] > 0 and d["unit"] == "GB/s" and d["higher_is_better"] is True
    assert d["steps"] == 1 and d["warmup"] == 3 and d["n_gpus"] == 1
    assert d["config"]["workload"] == "gemma2b_decode"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": "GB/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}


def test_fewer_than_three_warmup_steps_is_refused():
    r = _run("--impl", "reference", "--steps", "1", "--warmup", "2", timeout=120)
    assert r.returncode == 2
    assert "--warmup must be >= 3" in r.stderr


def test_step_stats():
    assert bench.step_stats([3.0, 1.0, 2.0]) == {"median": 2.0, "min": 1.0, "max": 3.0, "steps": 3}
    assert bench.step_stats([4.0, 1.0, 2.0, 3.0])["median"] == 2.5
    assert bench.step_stats([7.5]) == {"median": 7.5, "min": 7.5, "max": 7.5, "steps": 1}


@pytest.mark.parametrize("name", sorted(bench.WORKLOADS))
def test_every_workload_streams_weights_from_hbm(name):
    """Each timed step reads more distinct weight bytes than twice the L2, in the same
    order every pass, so no bench line is served from L2."""
    ws = bench.WORKLOADS[name]()
    distinct = bench.distinct_weight_bytes(ws)
    assert distinct > 2 * bench.L2_BYTES
    assert not bench.l2_policy(distinct).startswith("weights partly")


def test_distinct_bytes_count_reused_weights_once():
    import workloads as wl
    w = wl.action_expert_fused()
    assert bench.distinct_weight_bytes([w]) * 10 == w.weight_bytes()


def test_default_line_covers_every_configuration():
    """The default run's `configs` section has one entry per workload configuration (the
    single linear, the 2B decoder at M = 1, the action expert at M = 50, the 2B prefill and
    the vision tower, the 7B backbone at M = 1 and M = 280), each a bench workload."""
    keys = [k for k, _ in bench.CONFIG_WORKLOADS]
    assert sorted({k.split("_")[0] for k in keys}) == ["1", "2", "3", "4", "5"]
    for _, name in bench.CONFIG_WORKLOADS:
        assert name in bench.WORKLOADS
    Ms = {name: bench.WORKLOADS[name]()[0].M for _, name in bench.CONFIG_WORKLOADS}
    assert Ms == {"single_linear": 1, "gemma2b_decode": 1, "action_expert": 50,
                  "gemma2b_prefill": 816, "vit": 768, "llama7b_decode": 1, "llama7b_prefill": 280}
