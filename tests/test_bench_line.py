"""bench.py's JSON line on a GPU: every key of the benchmark contract, on a 4-layer slice
of the Llama-2-70B GQA shape (inputs larger than L2) and on the GPT-2-small shape
(inputs that fit in L2, so every timed step is preceded by an L2 flush)."""

import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench(*args, timeout=600):
    out = subprocess.run([sys.executable, "bench.py", *args], cwd=ROOT, capture_output=True, text=True,
                         timeout=timeout)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [ln for ln in out.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, out.stdout[-2000:]
    return json.loads(lines[0])


@pytest.mark.gpu
def test_bench_line_has_every_contract_key():
    j = _bench("--layers", "4", "--steps", "3", "--warmup", "3", "--cpu-seconds", "1")
    assert j["metric"].startswith("full-model sigma+scale refresh ms")
    assert j["unit"] == "ms" and j["higher_is_better"] is False
    assert j["n_gpus"] == 1 and j["steps"] == 3 and j["warmup"] == 3
    assert j["value"] > 0 and j["ms_per_step"] == j["value"]
    assert j["scaling"] == "weak" and j["vs_baseline"] is None and j["data"] == "synthetic"
    cfg = j["config"]
    assert cfg["workload"] == "llama2-70b-gqa" and cfg["layers"] == 4 and cfg["iters"] == 30
    assert "no flush needed" in cfg["l2"]
    r = j["roofline"]
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and r["kernel"] == "gram_fused"
    assert r["peak"] > 0 and abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-9
    # algorithmic bytes of the Gram launch: every W^Q_h and W^K_g once + the fp32 start vectors
    assert r["algorithmic_bytes"] == 4 * ((64 + 8) * 128 * 8192 * 2 + 64 * 8192 * 4)
    assert j["launches_per_step"] == 2 and j["gpu_launches"] == 2 * 3
    assert set(j["kernels_ms_per_step"]) == {"gram_fused", "writeback"}
    e = j["e2e"]
    assert e["unit"] == "ms" and e["value"] > j["value"]
    assert e["h2d_bytes_per_step"] == 4 * ((64 + 8) * 128 * 8192 * 2 + 64 * 8192 * 4)
    assert e["d2h_bytes_per_step"] == 4 * (4 * 64 + 4 + 4 * 64 * 8192)
    c = j["cpu_baseline"]
    assert c["kind"] == "oracle" and c["cores"] >= 1 and c["value"] > 0 and c["sample"]
    assert {"sm_mhz", "sm_max_mhz", "reasons"} <= set(j["clocks"])


@pytest.mark.gpu
def test_bench_flushes_l2_for_inputs_that_fit():
    j = _bench("--workload", "gpt2-small", "--steps", "3", "--warmup", "3", "--no-e2e", "--no-cpu-baseline")
    assert j["config"]["workload"] == "gpt2-small"
    assert "flush before every timed step" in j["config"]["l2"]
    assert j["value"] > 0 and j["gpu_launches"] == 2 * 3
    assert j["e2e"] is None and j["cpu_baseline"] is None
