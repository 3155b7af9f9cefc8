"""The reference arm of bench.py on CPU: it times the oracle on a bounded sample of the workload and
prints one JSON line with the same metric, unit and direction as the GPU arm."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_one_contract_line():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "0"], cwd=ROOT, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == "GB/s" and d["higher_is_better"] is True
    assert d["n_gpus"] == 1 and d["steps"] == 1 and d["warmup"] == 0
    assert d["value"] > 0 and d["e2e"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1 and cb["sample"]
    assert "workload" in d["config"]


def test_sweep_reports_a_failing_configuration_and_carries_on(monkeypatch):
    """run_sweep on CPU with every configuration replaced by a stub: a configuration that raises is
    reported under its own key as an error, and every later configuration still runs."""
    import types

    import torch

    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setattr(torch.cuda, "current_device", lambda: 0)
    monkeypatch.setattr(torch.cuda, "current_stream", lambda: None)
    monkeypatch.setattr(torch.cuda, "empty_cache", lambda: None)
    monkeypatch.setattr(bench, "l2_bytes", lambda dev: 129 << 20)
    ran = []

    def stub(name, fail=False):
        def f(*a, **k):
            ran.append(name)
            if fail:
                raise RuntimeError("planted")
            return {"ok": name}
        return f
    monkeypatch.setattr(bench, "sweep_config", stub("config"))
    monkeypatch.setattr(bench, "sweep_reuse", stub("reuse", fail=True))
    monkeypatch.setattr(bench, "sweep_quant", stub("quant"))
    monkeypatch.setattr(bench, "sweep_anchor_search", stub("anchor_search"))
    monkeypatch.setattr(bench, "sweep_anchor_residual", stub("anchor_residual"))
    out = bench.run_sweep(types.SimpleNamespace(reuse_batches=16), 6686.8)
    assert out["reuse"] == {"error": "RuntimeError: planted"}
    assert ran == ["config"] * 5 + ["reuse", "quant", "anchor_search", "anchor_residual"]
    assert set(out) == {"llama1", "qwen_kappa0.10", "qwen_kappa0.20", "qwen_kappa0.30",
                        "qwen_kappa0.50", "reuse", "llama32_quantized", "joint_anchor_search",
                        "joint_anchor_residual"}
