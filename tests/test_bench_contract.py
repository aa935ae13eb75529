"""The benchmark's output contract, checked on the CPU: the reference arm's
JSON line (the oracle timed on host cores), its silence on ranks other than
0, the algorithmic byte counts the roofline divides, and the option checks."""
import json
import os
import subprocess
import sys

import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _run(args, env=None):
    e = dict(os.environ)
    e.update(env or {})
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT, env=e,
                          capture_output=True, text=True, timeout=600)


def test_reference_arm_line():
    out = _run(["--impl", "reference", "--config", "tiny", "--steps", "2", "--warmup", "1"])
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC
    assert d["unit"] == "ms" and d["higher_is_better"] is False and d["vs_baseline"] is None
    assert d["n_gpus"] == 1 and d["steps"] == 2 and d["warmup"] == 1
    assert d["value"] > 0 and d["ms_per_step"] == d["value"]
    assert d["data"] == "synthetic" and d["config"]["workload"].startswith("tiny:")
    w = synth.CONFIGS["tiny"]
    assert d["config"] == bench.run_config(w, w.n_slabs, 1, 1, 1)  # the GPU arm's config object
    cpu = d["cpu_baseline"]
    assert cpu["kind"] == "oracle" and cpu["cores"] >= 1 and cpu["value"] == d["value"]
    assert cpu["sample"].startswith("every one of the 2 slabs")  # measured whole passes
    assert d["e2e"] == {"value": d["value"], "unit": "ms", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}


def test_reference_arm_is_silent_on_other_ranks():
    out = _run(["--impl", "reference", "--config", "tiny", "--steps", "1", "--warmup", "1"],
               env={"RANK": "1", "WORLD_SIZE": "2", "LOCAL_RANK": "1"})
    assert out.returncode == 0, out.stderr[-2000:]
    assert not [l for l in out.stdout.splitlines() if l.startswith("{")]


def test_pass_bytes_are_the_design_contract():
    """B = S D s (2N + 4C) + 4 S C: every K and V row read once by the scan,
    the kept rows read and written, the kept indices written."""
    w = synth.CONFIGS["llava"]
    r = 6
    pass_bytes, tight, per = bench.bytes_model(w, w.n_slabs, r)
    S, D, s, N, C, p = w.n_slabs, w.head_dim, 2, w.n_tokens, w.budget, w.p
    assert pass_bytes == S * D * s * (2 * N + 4 * C) + 4 * S * C == 1261625344
    assert tight == pass_bytes - S * D * s * r * p           # the recent rows' V is not needed
    assert per["gather"] == S * (4 * C * D * s + 4 * C) == 722132992
    assert per["score"] == S * (2 * (N - r * p) * D * s + 8 * (N - r * p))
    u = w.scaled(ablation="uniform")
    ub, ut, uper = bench.bytes_model(u, u.n_slabs, r)
    assert ub == ut == S * D * s * 4 * C + 4 * S * C             # Uniform Select reads no score
    assert uper["score"] == uper["recent_mean"] == 0


def test_ablation_needs_a_per_head_raw_van_workload():
    for cfg in ("llava_pool", "llava_shared"):
        out = _run(["--config", cfg, "--ablation", "uniform"])
        assert out.returncode == 2 and "--ablation" in out.stderr


def test_workload_strings_fit_the_record():
    """The driver's record keeps 120 characters of config.workload."""
    for w in synth.CONFIGS.values():
        assert len(bench.workload_desc(w)) <= 120, w.name


def test_traffic_is_reported_only_for_the_captured_sources(monkeypatch):
    """The roofline's DRAM traffic comes from the committed ncu capture only
    while the kernel sources are the ones it was taken on (their digest is
    stored beside it), and only for its own workload."""
    with open(os.path.join(ROOT, "profiles", "dram_traffic.json")) as fh:
        rec = json.load(fh)
    captured = rec["kernels"]["gather"]["dram_bytes_per_launch_full_size"]
    monkeypatch.setattr(bench, "source_digest", lambda: rec["source_digest"])
    assert bench.ncu_traffic("gather", rec["workload"]) == captured
    assert bench.ncu_traffic("gather", "qwen") is None
    assert bench.ncu_traffic("no_such_kernel", rec["workload"]) is None
    monkeypatch.setattr(bench, "source_digest", lambda: "0" * 16)
    assert bench.ncu_traffic("gather", rec["workload"]) is None
