"""The benchmark's reference arm (the oracle on the host cores) on the small
workload, run as the driver runs it: one JSON line with the GPU arm's config,
metric and unit, an oracle cpu_baseline and an e2e record without copies."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_line_on_the_small_workload():
    sys.path.insert(0, ROOT)
    import bench
    from paper_2607_29221_gb300 import workloads as wl
    env = dict(os.environ)
    env.pop("WORLD_SIZE", None)
    env.pop("RANK", None)
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload",
                        "single_64x256x128", "--steps", "2", "--warmup", "1"], capture_output=True, text=True,
                       timeout=600, env=env, cwd=ROOT)
    assert r.returncode == 0, r.stderr
    line = json.loads(r.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC and line["unit"] == "tokens/s"
    assert line["config"] == bench._config(wl.WORKLOADS["single_64x256x128"], 1)
    assert line["value"] > 0 and line["higher_is_better"] is True
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == line["value"] and cb["sample"]
    assert line["e2e"] == {"value": line["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}


def test_default_workload_is_the_decoder_layer():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.DEFAULT_WORKLOAD == "decoder_70b_prefill_2048"
    cfg = bench._config(__import__("paper_2607_29221_gb300.workloads", fromlist=["x"]).WORKLOADS[
        bench.DEFAULT_WORKLOAD], 1)
    assert cfg["l"] == 2048 and [x["m"] for x in cfg["linears"]] == [10240, 8192, 57344, 8192]
