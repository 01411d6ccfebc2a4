"""Host logic of bench.py that needs no GPU: the two arms report the same
config, the DRAM-traffic figure is dropped once the kernel source it was
captured on has changed, the count-rule ablations carry the paper's
thresholds, and the reference arm (the oracle on the host cores) prints
its contract line."""
import importlib
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    if ROOT not in sys.path:
        sys.path.insert(0, ROOT)
    return importlib.import_module("bench")


def test_both_arms_share_the_config(bench):
    from paper_2608_01784_gb300 import workloads as W
    # the stack: the GPU arm adds only its timing note to the shared dict
    c = bench.stack_config(1)
    assert c["workload"] == "llada_moe_stack16" and c["layers"] == 16
    assert c["tokens_per_step"] == 32 * 1024
    # single layers: one dict for both arms
    for name in ("llada_moe", "llada2_mini", "llada_moe_b32", "tiny_fp32"):
        lc = bench.layer_config(W.CONFIGS[name], 2)
        assert lc["workload"] == name and lc["tokens_per_step"] == W.CONFIGS[name].T
        assert lc["parallelism"] == "replicas2"


def test_traffic_follows_the_kernel_source(bench, monkeypatch):
    sha = bench.kernel_source_sha16()
    assert len(sha) == 16
    monkeypatch.setitem(bench.NCU_TRAFFIC, "x", (123, sha))
    assert bench.ncu_traffic("x") == 123
    monkeypatch.setitem(bench.NCU_TRAFFIC, "x", (123, "0" * 16))
    assert bench.ncu_traffic("x") is None          # captured on another source
    monkeypatch.setitem(bench.NCU_TRAFFIC, "x", (None, sha))
    assert bench.ncu_traffic("x") is None
    assert bench.ncu_traffic("no such workload") is None


def test_rule_ablations_use_the_paper_thresholds(bench):
    # App. B: Top-p 0.15 / 0.20 (LLaDA-MoE), 0.25 / 0.325 (LLaDA2.0-mini);
    # Expert-Threshold 0.0215 / 0.0190 and 0.0270 / 0.0220; counts in [1, 12]
    got = {n: o for n, o in bench.rule_ablations("llada_moe")}
    assert got["top_p_low"]["rule_threshold"] == 0.15
    assert got["top_p_high"]["rule_threshold"] == 0.20
    assert got["expert_threshold_low"]["rule_threshold"] == 0.0215
    assert got["expert_threshold_high"]["rule_threshold"] == 0.0190
    got = {n: o for n, o in bench.rule_ablations("llada2_mini")}
    assert got["top_p_high"]["rule_threshold"] == 0.325
    assert got["expert_threshold_low"]["rule_threshold"] == 0.0270
    for o in got.values():
        assert (o["k_min"], o["k_max"]) == (1, 12)
    assert bench.rule_ablations("tiny_fp32") == []


def test_traffic_key_ignores_comments_only(bench):
    a = "int f(int x) {  // twice\n  return 2 * x; /* no overflow\n here */ }\n"
    b = "// a header\nint f(int x) {\n    return 2 * x;\n}\n"
    c = "int f(int x) { return 3 * x; }"
    assert bench.code_of(a) == bench.code_of(b)
    assert bench.code_of(a) != bench.code_of(c)


def test_reference_arm_prints_the_contract_line(bench):
    # the reference arm (the oracle on the host cores) end to end on the tiny
    # layer: one JSON line with the GPU arm's config, metric and unit
    import json
    import subprocess
    from paper_2608_01784_gb300 import workloads as W
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--config",
                        "tiny_fp32", "--steps", "2", "--warmup", "1"],
                       cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC
    assert d["unit"] == "tokens/s" and d["higher_is_better"] is True
    assert d["steps"] == 2 and d["warmup"] == 1 and d["n_gpus"] == 1 and d["value"] > 0
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"],
                        "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1
    assert d["config"] == bench.layer_config(W.CONFIGS["tiny_fp32"], 1)
