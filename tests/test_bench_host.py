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


def test_client_rooflines_count_the_work_of_the_7b_step():
    """Algorithmic work of the client kernels on the 7B attention projection
    (l = 512, n = m = 4096, Example 3.1 parameters): 315,776 ChaCha20 blocks,
    2 x 512 x 8192 x 80 gathered MACs in Init X and 2 x 4096 x 512 x 80 in the
    unmask, 20 x 512 x 8192 x 652 and 20 x 512 x 4096 x 652 product flops."""
    sys.path.insert(0, ROOT)
    import types
    import bench
    from paper_2607_29221_gb300 import mosaic as M
    proto = types.SimpleNamespace(params=M.default_params())
    layer = types.SimpleNamespace(m=4096, n_pad=4096)
    kt = {"init_x:initx_draw": (2, 2e-3 * 2), "init_x:pgather": (4, 4e-3 * 2),
          "unmask:pgather": (4, 4e-3 * 2), "init_x:ring_gemm_tc": (2, 2e-3 * 2),
          "unmask:ring_gemm_tc": (2, 2e-3 * 2)}
    rows = bench._client_rooflines(kt, 2, [layer], proto, 512, 1910.6, "measured", 2070.0)
    assert len(rows) == 5

    def row(text):
        return [r for r in rows if text in r["kernel"]][0]
    clk = 2070e6
    draw = row("initx_draw_kernel")
    assert abs(draw["achieved"] - 315_776 * 976 / 2e-6 / 1e12) < 0.01
    assert abs(draw["peak"] - round(152 * 64 * clk / 1e12, 3)) < 1e-9
    gx = row("Init X LPN")
    assert abs(gx["achieved"] - 2 * 512 * 8192 * 80 * 4 / 4e-6 / 1e9) < 0.01
    assert abs(gx["peak"] - round(152 * 128 * clk / 1e9, 3)) < 1e-9
    gu = row("unmask LPN")
    assert abs(gu["achieved"] - 2 * 4096 * 512 * 80 * 4 / 4e-6 / 1e9) < 0.01
    tcx = row("Init X: R")
    assert abs(tcx["achieved"] - 20 * 512 * 8192 * 652 / 2e-6 / 1e12) < 0.01
    tcu = row("unmask: Y'")
    assert abs(tcu["achieved"] - 20 * 512 * 4096 * 652 / 2e-6 / 1e12) < 0.01
    assert all(abs(r["frac"] / (r["achieved"] / r["peak"]) - 1) < 1e-3 for r in rows)


def test_client_rooflines_take_the_measured_peaks():
    """With the device's measured ChaCha20 mix rate and shared-memory read rate
    the draw and gather rows use them as their peaks (and say so); the tensor
    rows keep the bf16 figure."""
    sys.path.insert(0, ROOT)
    import types
    import bench
    from paper_2607_29221_gb300 import mosaic as M
    proto = types.SimpleNamespace(params=M.default_params())
    layer = types.SimpleNamespace(m=4096, n_pad=4096)
    kt = {"init_x:initx_draw": (2, 4e-3), "init_x:pgather": (4, 8e-3), "unmask:pgather": (4, 8e-3),
          "init_x:ring_gemm_tc": (2, 4e-3), "unmask:ring_gemm_tc": (2, 4e-3)}
    rows = bench._client_rooflines(kt, 2, [layer], proto, 512, 1910.6, "measured", 2070.0,
                                   alu_measured=29.088e12, smem_measured=39794.3e9)
    by = {r["kernel"].split(" (")[0] + ":" + r["bound"]: r for r in rows}
    assert abs(by["initx_draw_kernel:alu"]["peak"] - 29.088) < 1e-9
    assert "mosaic_int_mix_rate" in by["initx_draw_kernel:alu"]["peak_source"]
    gathers = [r for r in rows if r["bound"] == "smem"]
    assert len(gathers) == 2
    assert all(abs(r["peak"] - 39794.3) < 1e-6 and "mosaic_smem_read_rate" in r["peak_source"] for r in gathers)
    assert all(r["peak"] == 1910.6 for r in rows if r["bound"] == "tensor")
